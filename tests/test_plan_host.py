"""Host-side invariants of the shared plan (csrc/bgpo_plan.h): the workspace
layout under every flag combination, the dX split-K choice against the split
buffer, and the clamping of the dW pairing offsets.

The header is compiled as plain C++ (g++) into a small program that prints the
plan for a grid of shapes; the checks below restate what the layout and the
split choice must satisfy, independently of how the header computes them.
"""
import json
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(os.path.dirname(HERE), "paper_2510_11683_gb300", "csrc")

PROGRAM = r"""
#include <cstdio>
#include <initializer_list>
#include "bgpo_plan.h"
using namespace bgpo;

static void layout(int64_t B, int64_t R, int64_t H, int64_t V) {
  const Geometry g = make_geometry(B, 1, R, H, V);
  for (int keep = 0; keep < 2; ++keep)
    for (int pair = 0; pair < 2; ++pair) {
      const Geometry gp = make_geometry(B, 1, R, H, V, 0, pair);
      const WsLayout L = make_ws_layout(gp, keep, pair);
      printf("{\"kind\": \"layout\", \"B\": %lld, \"R\": %lld, \"H\": %lld, \"V\": %lld, "
             "\"keep\": %d, \"pair\": %d, \"off\": [%zu, %zu, %zu, %zu, %zu, %zu, %zu, %zu, %zu, "
             "%zu, %zu, %zu, %zu, %zu, %zu], \"dz_rows\": %zu, \"dxp_elems\": %zu, "
             "\"zc_bytes\": %zu, \"total\": %zu, \"cap\": %lld, \"fwd\": %zu, \"m_pad\": %lld, "
             "\"n_vt\": %lld, \"dz_cols\": %zu, \"local\": %d, \"vc\": %lld, \"n_vc\": %lld, "
             "\"kb_vc_min\": %lld}\n",
             (long long)B, (long long)R, (long long)H, (long long)V, keep, pair, L.err, L.t,
             L.tnum, L.seg_off, L.rows, L.tgt, L.tgt_logit, L.lse, L.logp, L.part, L.xm, L.xmT,
             L.dz, L.dxp, L.zc, L.dz_rows, L.dxp_elems, L.zc_bytes, L.total,
             (long long)dxp_row_block_cap(gp), L.fwd_bytes, (long long)gp.m_pad,
             (long long)gp.n_vt, L.dz_cols, (int)L.dz_chunk_local, (long long)gp.vc,
             (long long)gp.n_vc, (long long)gp.kb_vc_min);
    }
  const int64_t cap = dxp_row_block_cap(g);
  for (int64_t mb = 1; mb <= g.m_pad / kPairM; ++mb)
    for (int pairs : {1, 7, 76}) {
      const int s = dx_splits(mb, dx_tiles_n(g.tiles_h), pairs, g.kb_v, cap);
      printf("{\"kind\": \"split\", \"mb\": %lld, \"tiles_n\": %lld, \"pairs\": %d, \"kb\": %lld, "
             "\"cap\": %lld, \"s\": %d, \"tiles_h\": %lld}\n",
             (long long)mb, (long long)dx_tiles_n(g.tiles_h), pairs, (long long)g.kb_v,
             (long long)cap, s, (long long)g.tiles_h);
    }
  for (int pair = 0; pair < 2; ++pair) {
    const WsLayout L = make_ws_layout(g, false, pair);
    for (int32_t stored : {-5, -1, 0, 1, 63, 64, 65, 1000, 4096, 1 << 20, 2147483647})
      printf("{\"kind\": \"roff\", \"dz_rows\": %zu, \"m_pad\": %lld, \"stored\": %d, "
             "\"off\": %lld}\n",
             L.dz_rows, (long long)g.m_pad, stored,
             (long long)row_offset(stored, (int64_t)L.dz_rows, g.m_pad));
  }
}

int main() {
  const long long shapes[][4] = {{2, 32, 64, 512},      {3, 301, 192, 1000},
                                 {5, 130, 320, 777},    {1, 1, 64, 1},
                                 {8, 256, 4096, 126464}, {16, 512, 4096, 126464},
                                 {32, 1024, 3584, 152064}, {4096, 1024, 64, 96}};
  for (const auto& s : shapes) layout(s[0], s[1], s[2], s[3]);
  for (int32_t j : {0, 1, 2, 15, 16, 1000, 65534, 65535})
    printf("{\"kind\": \"tag\", \"j\": %d, \"tag\": %d}\n", j, pend_tag(j));
  // row groups of the forward / dZ GEMMs: every tile exactly once
  for (int64_t H : {64, 3584, 4096, 16384})
    for (int64_t tm : {1, 2, 3, 17, 25, 26, 28, 32, 64, 129})
      for (int64_t tn : {1, 7, 494}) {
        const int64_t G = xm_row_groups(tm, H);
        static int seen[129 * 494];
        for (int64_t i = 0; i < tm * tn; ++i) seen[i] = 0;
        long long bad = 0, prev_n = -1, runs = 0;
        for (int64_t u = 0; u < tm * tn; ++u) {
          int64_t m, n;
          row_group_tile(u, tm, tn, G, &m, &n);
          if (m < 0 || m >= tm || n < 0 || n >= tn) { ++bad; continue; }
          ++seen[m * tn + n];
          if (n != prev_n) { ++runs; prev_n = n; }
        }
        long long once = 0;
        for (int64_t i = 0; i < tm * tn; ++i) once += seen[i] == 1;
        printf("{\"kind\": \"group\", \"H\": %lld, \"tm\": %lld, \"tn\": %lld, \"G\": %lld, "
               "\"bad\": %lld, \"once\": %lld, \"runs\": %lld}\n",
               (long long)H, (long long)tm, (long long)tn, (long long)G, bad, once, runs);
      }
  return 0;
}
"""


@pytest.fixture(scope="module")
def plan(tmp_path_factory):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    d = tmp_path_factory.mktemp("plan")
    src = d / "plan.cc"
    src.write_text(PROGRAM)
    exe = d / "plan"
    subprocess.run([cxx, "-std=c++17", "-O1", "-I", CSRC, str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout
    recs = [json.loads(line) for line in out.splitlines()]
    return {k: [r for r in recs if r["kind"] == k] for k in ("layout", "split", "roff", "tag", "group")}


def _ceil(a, b):
    return -(-a // b)


def test_workspace_regions_fit_in_order(plan):
    names = ["err", "t", "tnum", "seg_off", "rows", "tgt", "tgt_logit", "lse", "logp", "part",
             "xm", "xmT", "dz", "dxp", "zc"]
    for L in plan["layout"]:
        B, R, H, V = L["B"], L["R"], L["H"], L["V"]
        m_cap = B * R
        m_pad = _ceil(m_cap, 256) * 256
        v_pad = _ceil(V, 64) * 64
        n_vt = _ceil(V, 256)
        dz_rows = (2 if L["pair"] else 1) * m_pad
        assert L["dz_rows"] == dz_rows
        need = {"err": 64, "t": 4 * B, "tnum": 8 * B, "seg_off": 4 * (B + 1), "rows": 4 * m_cap,
                "tgt": 4 * m_pad, "tgt_logit": 4 * m_pad, "lse": 4 * m_pad, "logp": 4 * m_pad,
                "part": 8 * m_pad * n_vt, "xm": 2 * m_pad * H, "xmT": 2 * H * dz_rows,
                "dz": 2 * dz_rows * L["dz_cols"], "dxp": 4 * L["dxp_elems"],
                "zc": 4 * m_pad * v_pad if L["keep"] else 0}
        # the split buffer holds cap row blocks of 256 rows x H
        assert L["dxp_elems"] == L["cap"] * 256 * H
        off = dict(zip(names, L["off"]))
        order = [n for n in names if n != "zc" or L["keep"]]
        ends = [off[n] for n in order[1:]] + [L["total"]]
        for n, end in zip(order, ends):
            assert off[n] % 1024 == 0, (n, L)
            assert end - off[n] >= need[n], (n, L)
        assert L["zc_bytes"] == need["zc"]
        if not L["keep"]:
            assert off["zc"] == 0


def test_regions_up_to_xm_do_not_move_with_the_flags(plan):
    by_shape = {}
    for L in plan["layout"]:
        by_shape.setdefault((L["B"], L["R"], L["H"], L["V"]), []).append(L)
    for shape, ls in by_shape.items():
        prefixes = {tuple(L["off"][:11]) for L in ls}   # err .. xm
        assert len(prefixes) == 1, shape
        lean = [L for L in ls if not L["keep"] and not L["pair"]][0]
        assert all(L["total"] >= lean["total"] for L in ls)


def test_dx_split_choice(plan):
    for r in plan["split"]:
        mb, tn, pairs, kb, cap, s = r["mb"], r["tiles_n"], r["pairs"], r["kb"], r["cap"], r["s"]
        # dX tiles are 256 x 512: two 256-column blocks of H each
        assert tn == _ceil(r["tiles_h"], 2), r
        smax = max(1, min(16, kb, cap // mb))
        assert 1 <= s <= smax, r
        assert s == 1 or s * mb <= cap, r
        ideal = mb * tn / pairs
        t = lambda k: _ceil(mb * tn * k, pairs) / k
        if t(s) > 1.08 * ideal:      # nothing within 8%: the best count up to smax
            assert all(t(s) <= t(k) + 1e-12 for k in range(1, smax + 1)), r
        else:                        # the smallest count within 8%
            assert all(t(k) > 1.08 * ideal for k in range(1, s)), r


def test_split_room_allows_three_splits_at_the_largest_row_count(plan):
    for L in plan["layout"]:
        mb_max = _ceil(L["B"] * L["R"], 256)
        assert L["cap"] >= max(3 * mb_max, 16)


def test_pairing_offsets_are_clamped(plan):
    for r in plan["roff"]:
        room = r["dz_rows"] - r["m_pad"]
        off = r["off"]
        assert 0 <= off <= room and off % 64 == 0, r
        if 0 <= r["stored"] <= room:
            assert off == r["stored"] // 64 * 64, r
    assert {r["off"] for r in plan["roff"] if r["dz_rows"] == r["m_pad"]} == {0}


def test_pending_tags_are_not_small_integers(plan):
    for r in plan["tag"]:
        tag = r["tag"]
        assert tag != -1 and not (0 <= tag < 65536), r
        assert (tag & 0xFFFF) == r["j"] and (tag >> 16) == 0x5EED, r


def test_forward_regions_fit_the_documented_bound(plan):
    # bgpo_elbo_fwd_noalloc needs the forward regions only; include/bgpo.h
    # bounds them by roundup(B R, 256) (2 H + 8 ceil(V / 256) + 20) + 16 B + 12288
    for L in plan["layout"]:
        m_pad = -(-L["B"] * L["R"] // 256) * 256
        assert L["m_pad"] == m_pad
        bound = m_pad * (2 * L["H"] + 8 * -(-L["V"] // 256) + 20) + 16 * L["B"] + 12288
        assert L["off"][10] < L["fwd"] <= bound           # xm starts below the end
        assert L["fwd"] == L["off"][11]                    # Xm^T starts where it ends
        assert L["fwd"] % 1024 == 0


def test_vocabulary_chunks(plan):
    # default chunks: V split evenly into ceil(V / 32768) pieces rounded up to
    # 256 columns (one piece: the whole vocabulary, roundup(V, 64)); one chunk
    # with dW pairing or when the whole vocabulary's dZ fits 1 GiB; dZ holds one
    # chunk unless it must hold them all
    for L in plan["layout"]:
        V = L["V"]
        v_pad = _ceil(V, 64) * 64
        n = _ceil(V, 32768)
        w = _ceil(_ceil(V, n), 256) * 256
        small = 2 * L["m_pad"] * v_pad <= 1 << 30      # whole-vocabulary dZ within 1 GiB
        vc = v_pad if (L["pair"] or small or w >= V) else w
        assert L["vc"] == vc and L["n_vc"] == _ceil(V, vc)
        assert (L["n_vc"] - 1) * vc < V <= L["n_vc"] * vc
        last = V - (L["n_vc"] - 1) * vc
        assert L["kb_vc_min"] == _ceil(min(last, vc), 64)
        assert L["local"] == int(L["n_vc"] > 1 and not L["pair"])
        assert L["dz_cols"] == (vc if L["local"] else v_pad)
        assert vc % 256 == 0 or vc == v_pad


def test_row_groups_cover_every_tile_once(plan):
    for r in plan["group"]:
        tm, tn, G, H = r["tm"], r["tn"], r["G"], r["H"]
        assert r["bad"] == 0 and r["once"] == tm * tn, r
        xm = tm * 256 * H * 2
        if xm <= 52 << 20 or tm == 1:
            assert G == 1, r
        else:
            # groups of at most 40 MB of Xm, never more groups than row blocks
            assert G == min(tm, _ceil(xm, 40 << 20)), r
        # a vocabulary tile's units are consecutive within each group
        assert r["runs"] == G * tn or tn == 1, r

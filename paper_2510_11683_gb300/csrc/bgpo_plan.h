// Workspace layout, tile geometry and work splitting shared by the host code
// and the kernels of the BGPO LM-head ELBO path.
#pragma once

#include <stddef.h>
#include <stdint.h>

#ifdef __CUDACC__
#define BGPO_HD __host__ __device__ __forceinline__
#else
#define BGPO_HD inline
#endif

namespace bgpo {

// ---- GEMM tile geometry ---------------------------------------------------------
// A pair of CTAs (a 2-CTA cluster) computes one 256 x 256 fp32 tile with
// tcgen05.mma.cta_group::2: each CTA holds 128 rows of A, 128 of the 256 B
// columns and 128 accumulator rows in its own TMEM.
constexpr int kBM = 128;         // accumulator rows per CTA = TMEM lanes
constexpr int kPairM = 256;      // rows per pair tile
constexpr int kBN = 256;         // columns per tile = TMEM columns per accumulator
constexpr int kBNHalf = 128;     // B columns staged by each CTA of the pair
constexpr int kBK = 64;          // K per pipeline stage: one 128-byte swizzle row of bf16
constexpr int kUmmaK = 16;       // K of one tcgen05.mma kind::f16 instruction
constexpr int kStages = 6;       // TMA -> MMA pipeline depth
// The dX GEMM's tiles are kDxWide accumulators wide (256 x 512 for 2): each
// K block of A then feeds kDxWide MMAs, so the operand stream per flop into
// shared memory is 3/4 of a 256 x 256 tile's, and a wave of tiles covers all
// of H with half as many W column blocks re-read per row block. Both of the
// pair's 256-column accumulators hold one tile (the epilogue does not overlap
// the next tile's main loop), with kDxStages stages of 48 KB per CTA.
#ifndef BGPO_DX_WIDE
#define BGPO_DX_WIDE 2
#endif
constexpr int kDxWide = BGPO_DX_WIDE;
static_assert(kDxWide == 1 || kDxWide == 2, "dX tile width: one or two accumulators");
constexpr int kDxStages = kDxWide == 2 ? 4 : kStages;
constexpr int kMaxSplits = 16;   // split-K limit of the dX GEMM
// Widest vocabulary chunk of the backward by default: dZ is formed, used by
// the dX GEMM and the dW GEMM one chunk of at most this many columns at a
// time, so its buffer holds M x V_c instead of M x V.
constexpr int64_t kVChunkDefault = 32768;
// By default the vocabulary is walked in one piece when dZ for the whole of it
// takes at most this many bytes: chunks then save little memory and their
// launch tails cost most (few masked rows per launch).
constexpr int64_t kDzWholeMaxBytes = int64_t(1) << 30;

constexpr uint32_t kTileABytes = kBM * kBK * 2;       // 16 KB per CTA
constexpr uint32_t kTileBBytes = kBNHalf * kBK * 2;   // 16 KB per CTA
constexpr uint32_t kStageBytes = kTileABytes + kTileBBytes;
// Epilogue staging: each of the 4 epilogue warps double-buffers one 32-row x
// 128-byte sub-tile (32 fp32 or 64 bf16 columns) for its TMA stores.
constexpr uint32_t kEpiBufBytes = 32 * 128;
constexpr uint32_t kEpiBytes = 4 * 2 * kEpiBufBytes;   // 32 KB

// ---- kernel ids (trace + device error "where") --------------------------------
enum KernelId : int32_t {
  KID_MASK_COMPACT = 0,
  KID_GATHER = 1,
  KID_LMHEAD_FWD = 2,
  KID_LSE_COMBINE = 3,
  KID_SEQ_REDUCE = 4,
  KID_BOUND_COEFFS = 5,
  KID_LMHEAD_DZ = 6,
  KID_DX_GEMM = 7,
  KID_DX_REDUCE = 8,
  KID_DW_GEMM = 9,
  KID_GROUP_ADV = 10,
  KID_SELFTEST_WAIT = 11,
  KID_VRPO_COEFFS = 12,
  KID_DZ_FROM_LOGITS = 13,
  KID_XM_TRANSPOSE = 14,
  KID_COUNT = 15
};

BGPO_HD int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
BGPO_HD int64_t round_up(int64_t a, int64_t b) { return ceil_div(a, b) * b; }

// Column tiles of the dX GEMM for `tiles_h` hidden-size blocks of kBN columns.
BGPO_HD int64_t dx_tiles_n(int64_t tiles_h) { return ceil_div(tiles_h, kDxWide); }

// Row groups of the forward and dZ GEMMs. Consecutive tiles share a vocabulary
// tile of W, so every wave of tiles reads all of Xm's row blocks; once Xm
// outgrows what L2 keeps from one wave to the next (measured at the 8B head:
// no re-reads up to 36 MB, 3.5-5 reads per launch at 56-64 MB), the row blocks
// are walked in groups of at most kXmGroupBytes of Xm, each group over the
// whole vocabulary: W is then read once per group instead of Xm once per wave.
constexpr int64_t kXmGroupMinBytes = int64_t(52) << 20;
constexpr int64_t kXmGroupBytes = int64_t(40) << 20;
BGPO_HD int64_t xm_row_groups(int64_t tiles_m, int64_t H) {
  const int64_t bytes = tiles_m * kPairM * H * 2;
  if (tiles_m <= 1 || bytes <= kXmGroupMinBytes) return 1;
  const int64_t g = ceil_div(bytes, kXmGroupBytes);
  return g < tiles_m ? g : tiles_m;
}

// Tile (row block, vocabulary tile) of unit u of the forward and dZ GEMMs with
// `groups` row groups: group g holds row blocks [g tm / G, (g + 1) tm / G),
// its units follow those of the groups before it, and consecutive units of a
// group share a vocabulary tile.
BGPO_HD void row_group_tile(int64_t u, int64_t tiles_m, int64_t tiles_n, int64_t groups,
                            int64_t* m_blk, int64_t* n_blk) {
  int64_t g = 0;
  while (g + 1 < groups && ((g + 1) * tiles_m / groups) * tiles_n <= u) ++g;
  const int64_t r0 = g * tiles_m / groups;
  const int64_t rows = (g + 1) * tiles_m / groups - r0;
  const int64_t local = u - r0 * tiles_n;
  *n_blk = local / rows;
  *m_blk = r0 + local % rows;
}

// Split-K count of the dX GEMM (K = vocabulary) for `mb` pair row blocks times
// `tiles_n` column tiles on `num_pairs` CTA pairs: the smallest s whose
// wave-quantised time ceil(tiles*s/pairs)/s is within 8% of the ideal
// tiles/pairs, else the best s. s * mb never exceeds `row_block_cap`, which
// bounds the partial buffer independently of the SM count.
BGPO_HD int dx_splits(int64_t mb, int64_t tiles_n, int num_pairs, int64_t k_blocks,
                      int64_t row_block_cap) {
  const int64_t tiles_mn = mb * tiles_n;
  const int num_sms = num_pairs;
  if (tiles_mn <= 0 || num_sms <= 0) return 1;
  int64_t smax = kMaxSplits;
  if (k_blocks < smax) smax = k_blocks > 0 ? k_blocks : 1;
  if (row_block_cap / mb < smax) smax = row_block_cap / mb > 0 ? row_block_cap / mb : 1;
  const double ideal = (double)tiles_mn / (double)num_sms;
  int best = 1;
  double best_t = 1e300;
  for (int s = 1; s <= smax; ++s) {
    const double t = (double)ceil_div(tiles_mn * s, num_sms) / (double)s;
    if (t <= ideal * 1.08) return s;
    if (t < best_t) { best_t = t; best = s; }
  }
  return best;
}

// Width of the backward's vocabulary chunks. `request` 0 asks for the
// default: one chunk when dW pairing keeps the whole vocabulary's dZ anyway or
// when that dZ (m_pad rows of roundup(V, 64) bf16 values) fits
// kDzWholeMaxBytes, else the V columns split into ceil(V / kVChunkDefault)
// chunks of equal width rounded up to a tile. A positive request is a multiple
// of kBN (the host validates it). A width of V or more is a single chunk.
BGPO_HD int64_t vocab_chunk_width(int64_t V, int64_t request, bool pair_dw, int64_t m_pad) {
  int64_t w;
  if (request > 0) {
    w = request;
  } else if (pair_dw || 2 * m_pad * round_up(V, 64) <= kDzWholeMaxBytes) {
    w = V;
  } else {
    const int64_t n = ceil_div(V, kVChunkDefault);
    w = round_up(ceil_div(V, n), kBN);
  }
  return w >= V ? round_up(V, 64) : w;
}

// Geometry derived from the problem sizes (host and device agree on it).
struct Geometry {
  int64_t B, P, R, H, V;
  int64_t m_cap;      // B * R: most masked rows a sample can have
  int64_t m_pad;      // m_cap rounded up to a pair tile of rows
  int64_t v_pad;      // V rounded up to 64 (row pitch of the kept logits)
  int64_t n_vt;       // vocabulary tiles of kBN columns
  int64_t tiles_h;    // hidden-size tiles of kBN columns
  int64_t kb_v;       // K blocks of kBK over the vocabulary
  int64_t vc;         // vocabulary chunk width of the backward (v_pad when one chunk)
  int64_t n_vc;       // vocabulary chunks: chunk c covers [c vc, min(V, (c + 1) vc))
  int64_t kb_vc_min;  // K blocks of kBK of the narrowest chunk (the dX split bound)
};

BGPO_HD Geometry make_geometry(int64_t B, int64_t P, int64_t R, int64_t H, int64_t V,
                               int64_t vchunk_request = 0, bool pair_dw = false) {
  Geometry g;
  g.B = B; g.P = P; g.R = R; g.H = H; g.V = V;
  g.m_cap = B * R;
  g.m_pad = round_up(g.m_cap, kPairM);
  g.v_pad = round_up(V, 64);
  g.n_vt = ceil_div(V, kBN);
  g.tiles_h = ceil_div(H, kBN);
  g.kb_v = ceil_div(V, kBK);
  g.vc = vocab_chunk_width(V, vchunk_request, pair_dw, g.m_pad);
  g.n_vc = ceil_div(V, g.vc);
  const int64_t last = V - (g.n_vc - 1) * g.vc;
  g.kb_vc_min = ceil_div(last < g.vc ? last : g.vc, kBK);
  return g;
}

// Vocabulary range [v0, v1) of backward chunk c.
BGPO_HD int64_t chunk_begin(const Geometry& g, int64_t c) { return c * g.vc; }
BGPO_HD int64_t chunk_end(const Geometry& g, int64_t c) {
  const int64_t e = (c + 1) * g.vc;
  return e < g.V ? e : g.V;
}

// Device workspace layout. Every region starts on a 1024-byte boundary (TMA
// tiles with 128-byte swizzle want 1024-byte aligned bases).
struct WsLayout {
  size_t err;        // int32[16]: the fields of ErrField
  size_t t;          // float[B]    t_{b,j}
  size_t tnum;       // uint32[2B]  T numerator (t = T / D), (low, high) words
  size_t seg_off;    // int32[B+1]  first compacted row of each sequence
  size_t rows;       // int32[m_cap] b*R + i of each masked position, ascending
  size_t tgt;        // int32[m_pad] target token of each compacted row
  size_t tgt_logit;  // float[m_pad] z_{r, y_r}
  size_t lse;        // float[m_pad] log-sum-exp of each row's logits
  size_t logp;       // float[m_pad] log p(y_r)
  size_t part;       // float2[m_pad * n_vt] (max, sum-exp) per (row, vocab tile)
  size_t xm;         // bf16[m_pad * H] gathered masked hidden states
  size_t fwd_bytes;  // end of the regions a forward pass uses (err .. xm); the same under
                     // every flag
  size_t xmT;        // bf16[H * dz_rows] the same, transposed (the dW GEMM's K-major operand)
  size_t dz;         // bf16[dz_rows * dz_cols] dL/dz of the current sample (and of a pending
                     // one): one vocabulary chunk at a time, or the whole vocabulary
  size_t dz_rows;    // m_pad, or 2 m_pad when the dW GEMM pairs samples
  size_t dz_cols;    // vc when the buffer holds one chunk, v_pad when it holds them all
  bool dz_chunk_local;  // chunk c is formed at column 0 (else at column c vc)
  size_t dxp;        // float[dxp_elems] split-K partials of dX
  size_t dxp_elems;
  size_t zc;         // float[m_pad * v_pad] logits kept by the forward (last region)
  size_t zc_bytes;   // 0 when the forward keeps no logits
  size_t total;
};

BGPO_HD size_t align_ws(size_t x) { return (x + 1023) & ~(size_t)1023; }

// Pair row blocks (256 rows) the split-K partial buffer holds, which bounds the
// splits s of a sample with mb row blocks to s * mb <= cap: three splits at the
// largest mb, up to kMaxSplits for small mb (measured: a second split takes
// 6-8% off a dX GEMM whose unsplit tiles leave a last wave 20% full; with
// 256 x 512 tiles, room for a third split took 1.5% off the dX GEMMs of a
// step against room for two).
BGPO_HD int64_t dxp_row_block_cap(const Geometry& g) {
  const int64_t mb_max = g.m_pad / kPairM;
  const int64_t small = 4 * mb_max < 4 * kMaxSplits ? 4 * mb_max : 4 * kMaxSplits;
  int64_t cap = 3 * mb_max > small ? 3 * mb_max : small;
  return cap > kMaxSplits ? cap : kMaxSplits;
}

// `keep_logits` appends the fp32 logit region. `pair_dw` doubles the rows of
// dZ and the columns of Xm^T: the rows of an even sample wait there for the
// dW GEMM of the next sample, whose rows follow them; its dZ rows then span
// the whole vocabulary. Otherwise dZ holds one vocabulary chunk.
BGPO_HD WsLayout make_ws_layout(const Geometry& g, bool keep_logits, bool pair_dw) {
  WsLayout L;
  size_t o = 0;
  L.dz_rows = (pair_dw ? 2 : 1) * (size_t)g.m_pad;
  L.dz_chunk_local = !pair_dw && g.n_vc > 1;
  L.dz_cols = L.dz_chunk_local ? (size_t)g.vc : (size_t)g.v_pad;
  L.err = o;       o = align_ws(o + 64);
  L.t = o;         o = align_ws(o + 4 * (size_t)g.B);
  L.tnum = o;      o = align_ws(o + 8 * (size_t)g.B);
  L.seg_off = o;   o = align_ws(o + 4 * (size_t)(g.B + 1));
  L.rows = o;      o = align_ws(o + 4 * (size_t)g.m_cap);
  L.tgt = o;       o = align_ws(o + 4 * (size_t)g.m_pad);
  L.tgt_logit = o; o = align_ws(o + 4 * (size_t)g.m_pad);
  L.lse = o;       o = align_ws(o + 4 * (size_t)g.m_pad);
  L.logp = o;      o = align_ws(o + 4 * (size_t)g.m_pad);
  L.part = o;      o = align_ws(o + 8 * (size_t)g.m_pad * (size_t)g.n_vt);
  L.xm = o;        o = align_ws(o + 2 * (size_t)g.m_pad * (size_t)g.H);
  L.fwd_bytes = o;
  L.xmT = o;       o = align_ws(o + 2 * (size_t)g.H * L.dz_rows);
  L.dz = o;        o = align_ws(o + 2 * L.dz_rows * L.dz_cols);
  L.dxp_elems = (size_t)dxp_row_block_cap(g) * kPairM * (size_t)g.H;
  L.dxp = o;       o = align_ws(o + 4 * L.dxp_elems);
  L.zc_bytes = keep_logits ? 4 * (size_t)g.m_pad * (size_t)g.v_pad : 0;
  L.zc = keep_logits ? o : 0;
  o = align_ws(o + L.zc_bytes);
  L.total = o;
  return L;
}

// Indices into the int32 error word:
//   ERR_STATUS, ERR_WHERE  the device error (bgpo_get_device_error)
//   ERR_SAMPLE, ERR_M      the sample j the workspace holds and its masked rows
//   ERR_LOGITS    1 while the logit region holds the current sample's logits
//                 (set by the forward that wrote them, cleared by the masking of
//                 a new sample and by a forward that keeps none)
//   ERR_DX_SPLITS the split-K count the last dX GEMM used
//   ERR_PEND      pend_tag(j) while sample j's dZ and Xm^T rows wait for the dW
//                 GEMM of sample j + 1, else -1
//   ERR_PEND_OFF  the row at which sample j + 1's dZ and Xm^T rows start: M_j
//                 rounded up to a K block
//   ERR_ROW_OFF   set by the masking: the first dZ / Xm^T row of the current
//                 sample (ERR_PEND_OFF when it pairs with the pending sample,
//                 else 0)
//   ERR_PAIRED    set by the masking: 1 when the current sample pairs
//   ERR_DW_K0     set by the backward before its dW GEMM: the first K row that
//                 GEMM adds (0 while the partner is pending, ERR_ROW_OFF once
//                 an earlier backward of this sample has added the partner)
enum ErrField : int {
  ERR_STATUS = 0, ERR_WHERE = 1, ERR_SAMPLE = 2, ERR_M = 3, ERR_LOGITS = 4, ERR_DX_SPLITS = 5,
  ERR_PEND = 6, ERR_PEND_OFF = 7, ERR_ROW_OFF = 8, ERR_PAIRED = 9, ERR_DW_K0 = 10
};

// Tag of a pending sample (n_t < 2^16): neither -1 nor a small integer that
// memory not yet written by this library is likely to hold.
BGPO_HD int32_t pend_tag(int32_t j) { return (int32_t)(0x5EED0000u | (uint32_t)j); }

// First dZ / Xm^T row of the current sample, clamped to the room the layout
// has for a pending sample (none without pairing) and to a K block.
BGPO_HD int64_t row_offset(int32_t stored, int64_t dz_rows, int64_t m_pad) {
  const int64_t room = dz_rows - m_pad;
  int64_t off = stored < 0 ? 0 : (int64_t)stored;
  if (off > room) off = room;
  return off & ~(int64_t)(kBK - 1);
}

}  // namespace bgpo

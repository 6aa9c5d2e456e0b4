// The four LM-head contractions of the BGPO ELBO path on sm_103a tensor cores.
//
// Each is a persistent, warp-specialised kernel launched as 2-CTA clusters. A
// CTA pair computes 256 x 256 fp32 tiles with tcgen05.mma.cta_group::2: CTA r
// of the pair stages rows [128 r, 128 r + 128) of the A tile and columns
// [128 r, 128 r + 128) of the B tile, and holds accumulator rows
// [128 r, 128 r + 128) in its TMEM. The dX GEMM's tiles are kDxWide such
// tiles side by side, sharing their A tile. Roles in each CTA (192 threads):
//   warp 0      TMA producer: 128-byte-swizzled bf16 boxes into a 6-stage ring
//               of 32 KB (dX: 4 stages of 48 KB); every copy of both CTAs completes on the even CTA's
//               "full" barrier, which the even CTA alone arms with both CTAs'
//               transaction bytes (a negative transaction count in between is
//               allowed)
//   warp 1      TMEM allocation (pair, 512 columns = two accumulators); in the
//               even CTA also the MMA issuer (M = 256, N = 256, K = 16; the
//               dX GEMM issues one per accumulator of its tile)
//   warps 2-5   epilogue: tcgen05.ld of this CTA's accumulator rows, fused
//               per-kind epilogue, TMA stores / reductions from shared memory
// The epilogue of tile n overlaps the main loop of tile n+1, except in the dX
// GEMM when its tiles occupy both accumulators.
//
// Kinds (Xm = gathered masked hidden states [M, H], W = LM head [V, H]):
//   GEMM_FWD  z = Xm W^T; epilogue: online max / sum-exp per (row, vocab tile)
//             and the target logit (Eq. 4: log softmax gathered at y^i); when
//             the workspace has a logit region the fp32 tile also leaves
//             through TMA stores, for the backward.
//   GEMM_DZ   z = Xm W^T recomputed (when the forward kept no logits) for one
//             vocabulary chunk of the backward; epilogue: dz = w_r (onehot -
//             e^{z - lse}) stored as bf16 (gradient of Eq. 4 weighted by
//             Eq. 13's dL/dl).
//   GEMM_DX   dXm += dZ_c W_c (K = the chunk's vocabulary; 256 x 512 tiles): split-K partials in
//             fp32, stored by the first chunk and added by the later ones, or,
//             when the launch needs no split, added straight into the dX rows.
//   GEMM_DW   dW[chunk rows] += dZ_c^T Xm (K = masked rows; Xm read as its
//             transpose, so that the B operand is K-major), fp32 TMA
//             reduce-add. With dW pairing (whole-vocabulary dZ), K also covers
//             the rows of the pending sample before.
//
// Every wait is bounded (time and polls); a wait that runs out sets the
// workspace error word to BGPO_ERR_TIMEOUT and both CTAs drain and exit.
#include <math.h>

#include <mutex>

#include "bgpo_device.cuh"
#include "bgpo_internal.h"

namespace bgpo {

namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr int32_t kStatusInvalidArg = 1;  // BGPO_ERR_INVALID_ARG
constexpr int32_t kStatusTimeout = 8;     // BGPO_ERR_TIMEOUT
constexpr int kThreads = 192;             // 6 warps
constexpr uint32_t kTmemCols = 2 * kBN;   // two accumulators
constexpr uint32_t kMnChunkBytes = 64 * 64 * 2;   // one 64 x 64 bf16 TMA box (MN-major)
constexpr uint16_t kBothCtas = 0x3;

struct GemmParams {
  Geometry g;
  int num_pairs;
  int32_t j;
  int64_t v_begin, v_end, dz_col0, chunk;
  WsPtrs w;
  const float* coef;
  float* dW;
  float* dX;
  bool pair_consume;
};

struct Work {
  int64_t units, tiles_m, tiles_n, kb_total;
  int64_t kb_first;  // first K block (dW: a partner already added is skipped)
  int64_t groups;    // forward and dZ: row groups (xm_row_groups)
  int splits;
};

struct Unit {
  int32_t m_blk, n_blk, split, kb0, kb_n;
};

// `roff`: the first dZ / Xm^T row of the sample (dW pairing; 0 otherwise). The
// dW GEMM's K range [k0, roff + M) then covers a pending sample's rows too when
// k0 = 0.
template <int KIND>
__device__ __forceinline__ Work make_work(const GemmParams& p, int32_t M, int64_t roff,
                                          int64_t k0) {
  Work w;
  w.splits = 1;
  w.kb_first = 0;
  w.groups = 1;
  if (KIND == GEMM_FWD || KIND == GEMM_DZ) {
    w.tiles_m = ceil_div(M, kPairM);
    w.tiles_n = KIND == GEMM_FWD ? p.g.n_vt : ceil_div(p.v_end - p.v_begin, kBN);
    // a last K block past H reads the tensor maps' zero fill
    w.kb_total = ceil_div(p.g.H, kBK);
    w.units = w.tiles_m * w.tiles_n;
    w.groups = xm_row_groups(w.tiles_m, p.g.H);
  } else if (KIND == GEMM_DX) {
    w.tiles_m = ceil_div(M, kPairM);
    w.tiles_n = dx_tiles_n(p.g.tiles_h);
    w.kb_total = ceil_div(p.v_end - p.v_begin, kBK);
    // one split count for every chunk of the sample (the partials of split s
    // accumulate over the chunks), bounded by the narrowest chunk's K blocks
    w.splits = w.tiles_m > 0 ? dx_splits(w.tiles_m, w.tiles_n, p.num_pairs, p.g.kb_vc_min,
                                         dxp_row_block_cap(p.g))
                             : 1;
    w.units = w.tiles_m * w.tiles_n * w.splits;
  } else {  // GEMM_DW
    w.tiles_m = ceil_div(p.v_end - p.v_begin, kPairM);
    w.tiles_n = p.g.tiles_h;
    w.kb_total = ceil_div(roff + M, kBK);
    w.kb_first = k0 / kBK;
    w.units = w.kb_total > w.kb_first ? w.tiles_m * w.tiles_n : 0;
  }
  return w;
}

template <int KIND>
__device__ __forceinline__ Unit unit_of(const Work& w, int64_t u) {
  Unit t;
  t.split = 0;
  if (KIND == GEMM_FWD || KIND == GEMM_DZ) {
    // consecutive units share a vocabulary tile of W: it is read from HBM once
    // per row group
    int64_t m, n;
    row_group_tile(u, w.tiles_m, w.tiles_n, w.groups, &m, &n);
    t.m_blk = (int32_t)m;
    t.n_blk = (int32_t)n;
    t.kb0 = 0;
    t.kb_n = (int32_t)w.kb_total;
  } else if (KIND == GEMM_DX) {
    // consecutive units share a row block of dZ (measured 2% faster than
    // sharing a column block of W, and than grouped rasters)
    const int64_t per_split = w.tiles_m * w.tiles_n;
    t.split = (int32_t)(u / per_split);
    const int64_t rem = u % per_split;
    t.m_blk = (int32_t)(rem / w.tiles_n);
    t.n_blk = (int32_t)(rem % w.tiles_n);
    const int64_t k0 = (int64_t)t.split * w.kb_total / w.splits;
    const int64_t k1 = (int64_t)(t.split + 1) * w.kb_total / w.splits;
    t.kb0 = (int32_t)k0;
    t.kb_n = (int32_t)(k1 - k0);
  } else {
    // consecutive units share a vocabulary block of dZ^T
    t.m_blk = (int32_t)(u / w.tiles_n);
    t.n_blk = (int32_t)(u % w.tiles_n);
    t.kb0 = (int32_t)w.kb_first;
    t.kb_n = (int32_t)(w.kb_total - w.kb_first);
  }
  return t;
}

// Shared-memory plan of one kind: 6 pipeline stages and the epilogue's
// staging buffers (the forward GEMM stages its fp32 logits there when it keeps
// them).
template <int KIND>
struct Shape {
  static constexpr int nacc = KIND == GEMM_DX ? kDxWide : 1;  // accumulators per tile
  static constexpr int bufs = 2 / nacc;                        // tiles in TMEM at once
  static constexpr int stages = KIND == GEMM_DX ? kDxStages : kStages;
  static constexpr uint32_t b_bytes = nacc * kTileBBytes;      // B bytes per CTA and stage
};

template <int KIND>
struct SmemPlan {
  static constexpr int stages = Shape<KIND>::stages;
  static constexpr uint32_t epi_bytes = kEpiBytes;
  static constexpr uint32_t bytes =
      stages * (kTileABytes + Shape<KIND>::b_bytes) + epi_bytes + 1024 + 1024;
  static_assert(bytes <= 232448, "shared memory per CTA");
};

// Operand majorness: forward and dZ read Xm and W K-major; dX reads dZ K-major
// and W MN-major; dW reads dZ^T MN-major and Xm^T (a transposed copy) K-major.
// Four MN-major boxes per stage (dW on Xm itself) measured 12% slower.
template <int KIND>
struct Majors {
  static constexpr bool a_mn = (KIND == GEMM_DW);
  static constexpr bool b_mn = (KIND == GEMM_DX);
};

// Rows of the K-major B operand (W for forward and dZ, Xm^T for dW).
template <int KIND>
__device__ __forceinline__ int64_t b_rows(const GemmParams& p) {
  return KIND == GEMM_DW ? p.g.H : p.g.V;
}

// First row of the K-major B operand in this launch: dZ's W rows start at the
// chunk's first vocabulary entry.
template <int KIND>
__device__ __forceinline__ int64_t b_base(const GemmParams& p) {
  return KIND == GEMM_DZ ? p.v_begin : 0;
}

// Bytes this CTA's copies deliver for one stage of unit t (boxes that would lie
// wholly outside the operand are not issued; their MMA outputs are discarded).
template <int KIND>
__device__ __forceinline__ uint32_t stage_bytes(const GemmParams& p, const Unit& t, uint32_t rank) {
  const int64_t a0 = (int64_t)t.m_blk * kPairM + (int64_t)rank * kBM;
  const int64_t b0 =
      b_base<KIND>(p) + (int64_t)t.n_blk * Shape<KIND>::nacc * kBN + (int64_t)rank * kBNHalf;
  uint32_t bytes = 0;
  if (!Majors<KIND>::a_mn) {
    bytes += kTileABytes;
  } else {
    // dZ^T vocabulary columns of this CTA inside the dZ buffer
    for (int c = 0; c < kBM / 64; ++c)
      if (p.dz_col0 + a0 + c * 64 < p.w.dz_cols) bytes += kMnChunkBytes;
  }
  if (!Majors<KIND>::b_mn) {
    if (b0 < b_rows<KIND>(p)) bytes += kTileBBytes;
  } else {
    for (int g = 0; g < Shape<KIND>::nacc; ++g)
      for (int c = 0; c < kBNHalf / 64; ++c)
        if (b0 + g * kBN + c * 64 < p.g.H) bytes += kMnChunkBytes;
  }
  return bytes;
}

// Issues this CTA's TMA loads of one stage; they complete on `cbar`, the even
// CTA's full barrier (shared::cluster address). The dX GEMM's dZ rows start at
// `roff`; its K blocks count from the chunk's first vocabulary entry, which
// lies at dZ column dz_col0 and W row v_begin.
template <int KIND>
__device__ __forceinline__ void load_stage(const GemmParams& p, const CUtensorMap* ma,
                                           const CUtensorMap* mb, uint32_t sa, uint32_t sb,
                                           uint32_t cbar, const Unit& t, int32_t kb,
                                           uint32_t rank, int64_t roff) {
  const int32_t a0 =
      t.m_blk * kPairM + (int32_t)rank * kBM + (KIND == GEMM_DX ? (int32_t)roff : 0);
  const int64_t b0 =
      b_base<KIND>(p) + (int64_t)t.n_blk * Shape<KIND>::nacc * kBN + (int64_t)rank * kBNHalf;
  if (!Majors<KIND>::a_mn) {
    const int32_t ka = kb * kBK + (KIND == GEMM_DX ? (int32_t)p.dz_col0 : 0);
    tma_load_2d_pair(sa, ma, cbar, ka, a0);
  } else {
    // dZ^T rows of this CTA: 2 boxes of 64 vocabulary columns x 64 masked rows
#pragma unroll
    for (int c = 0; c < kBM / 64; ++c) {
      const int64_t xa = p.dz_col0 + a0 + c * 64;
      if (xa < p.w.dz_cols)
        tma_load_2d_pair(sa + c * kMnChunkBytes, ma, cbar, (int32_t)xa, kb * kBK);
    }
  }
  if (!Majors<KIND>::b_mn) {
    if (b0 < b_rows<KIND>(p)) tma_load_2d_pair(sb, mb, cbar, kb * kBK, (int32_t)b0);
  } else {
    // W columns of this CTA (GEMM_DX): 2 boxes of 64 x 64 per accumulator of the
    // tile (accumulator g's at sb + g * kTileBBytes), rows from the chunk's start
    const int32_t kw = (int32_t)(p.v_begin + (int64_t)kb * kBK);
#pragma unroll
    for (int g = 0; g < Shape<KIND>::nacc; ++g)
#pragma unroll
      for (int c = 0; c < kBNHalf / 64; ++c)
        if (b0 + g * kBN + c * 64 < p.g.H)
          tma_load_2d_pair(sb + g * kTileBBytes + c * kMnChunkBytes, mb, cbar,
                           (int32_t)(b0 + g * kBN + c * 64), kw);
  }
}

__device__ __forceinline__ float bits_f(uint32_t v) { return __uint_as_float(v); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// ---- epilogues: one thread per accumulator row; row0 = first row of the warp --------

// Epilogue staging of one warp: two 32-row x 128-byte buffers in the 128-byte
// swizzled layout the TMA tensor maps use (16-byte chunk q of row r stored at
// chunk q ^ (r & 7)), so that 32 lanes writing one row each hit 8 bank groups.
struct EpiStage {
  uint32_t base;   // shared address of this warp's first buffer (1024-aligned)
  int buf;         // buffer the next sub-tile goes to

  // Returns the shared address of a buffer free for writing: the bulk group
  // that last read it (two sub-tiles ago) has finished reading.
  __device__ __forceinline__ uint32_t acquire(int lane) {
    if (lane == 0) bulk_wait_group_read<1>();
    __syncwarp();
    return base + (uint32_t)buf * kEpiBufBytes;
  }
  // Hands the written buffer to lane 0, which issues the bulk copy `issue`.
  template <class Issue>
  __device__ __forceinline__ void release(int lane, uint32_t sbuf, Issue issue) {
    fence_proxy_async_shared();
    __syncwarp();
    if (lane == 0) {
      issue(sbuf);
      bulk_commit_group();
    }
    buf ^= 1;
  }
};

// Writes 8 16-byte chunks (one 128-byte row of the sub-tile) for row `lane`.
__device__ __forceinline__ void stage_row(uint32_t sbuf, int lane, const uint4 (&chunk)[8]) {
  const uint32_t row = sbuf + (uint32_t)lane * 128u;
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const uint32_t a = row + (uint32_t)((q ^ (lane & 7)) * 16);
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(chunk[q].x),
                 "r"(chunk[q].y), "r"(chunk[q].z), "r"(chunk[q].w)
                 : "memory");
  }
}

// GEMM_FWD: per (row, vocab tile) the pair (max z, sum e^{z - max}) and, in the
// tile holding y_r, the target logit z_{r, y_r}; with a logit region, the
// fp32 logits too (32-column sub-tiles through TMA stores into [m_pad, v_pad]).
__device__ __forceinline__ void epi_fwd(const GemmParams& p, const CUtensorMap* map_c, int32_t M,
                                        const Unit& t, int64_t row0, int lane, uint32_t tb,
                                        EpiStage& st) {
  const int64_t r = row0 + lane;
  const bool valid = r < M;
  const int32_t y = valid ? p.w.tgt[r] : -1;
  const int32_t v0 = t.n_blk * kBN;
  const int32_t V = (int32_t)p.g.V;
  float m = -INFINITY, s = 0.f, tl = 0.f;
  bool hit = false;
#pragma unroll 1
  for (int c = 0; c < kBN / 32; ++c) {
    const int32_t col0 = v0 + c * 32;
    if (col0 >= V) break;  // warp-uniform
    uint32_t raw[32];
    tmem_ld_32x32b_x32(tb + c * 32, raw);
    tmem_ld_wait();
    const int nvalid = min(32, V - col0);
    // the row's target lies in this sub-tile for about one sub-tile in 4000:
    // test it once instead of once per column
    if ((uint32_t)(y - col0) < 32u) {
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (col0 + k == y) { tl = bits_f(raw[k]); hit = true; }
    }
    float cm = -INFINITY;
    float acc = 0.f;
    float mn;
    if (nvalid == 32) {  // warp-uniform: every column lies inside the vocabulary
#pragma unroll
      for (int k = 0; k < 32; ++k) cm = fmaxf(cm, bits_f(raw[k]));
      mn = fmaxf(m, cm);
      const float mnl = mn * kLog2e;
#pragma unroll
      for (int k = 0; k < 32; ++k) acc += ex2_ftz(fmaf(bits_f(raw[k]), kLog2e, -mnl));
    } else {
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (k < nvalid) cm = fmaxf(cm, bits_f(raw[k]));
      mn = fmaxf(m, cm);
      const float mnl = mn * kLog2e;
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (k < nvalid) acc += ex2_ftz(fmaf(bits_f(raw[k]), kLog2e, -mnl));
    }
    s = s * ex2_ftz((m - mn) * kLog2e) + acc;
    m = mn;
    if (p.w.zc != nullptr) {  // kernel-uniform; col0 < V <= v_pad, both multiples of 32
      uint4 chunk[8];
#pragma unroll
      for (int q = 0; q < 8; ++q)
        chunk[q] = make_uint4(raw[4 * q], raw[4 * q + 1], raw[4 * q + 2], raw[4 * q + 3]);
      const uint32_t sbuf = st.acquire(lane);
      stage_row(sbuf, lane, chunk);
      st.release(lane, sbuf, [&](uint32_t a) { tma_store_2d(map_c, a, col0, (int32_t)row0); });
    }
  }
  if (valid) {
    p.w.part[r * p.g.n_vt + t.n_blk] = make_float2(m, s);
    if (hit) p.w.tgt_logit[r] = tl;
  }
}

// GEMM_DZ: dz_{r,v} = w_r (1[v = y_r] - e^{z_{r,v} - lse_r}) as bf16, zero for
// rows >= M and vocabulary columns >= V; 64-column sub-tiles leave through TMA
// stores into dZ [dz_rows, dz_cols], from row `roff` on; vocabulary entry v
// lands in column v - v_begin + dz_col0.
__device__ __forceinline__ void epi_dz(const GemmParams& p, const CUtensorMap* map_c, int32_t M,
                                       const Unit& t, int64_t row0, int64_t roff, int lane,
                                       uint32_t tb, EpiStage& st) {
  const int64_t r = row0 + lane;
  const bool valid = r < M;
  float w = 0.f, lse_l2 = 0.f;
  int32_t y = -1;
  if (valid && BGPO_IN_BOUNDS(p.w.err, p.w.rows[r] >= 0 && p.w.rows[r] < p.g.m_cap,
                              KID_LMHEAD_DZ * 16 + 10)) {
    const int32_t b = p.w.rows[r] / (int32_t)p.g.R;
    w = p.coef[b] / p.w.t[b];
    lse_l2 = p.w.lse[r] * kLog2e;
    y = p.w.tgt[r];
  }
  const int32_t v0 = (int32_t)p.v_begin + t.n_blk * kBN;
  const int32_t V = (int32_t)p.g.V;
  const int32_t shift = (int32_t)(p.dz_col0 - p.v_begin);   // vocabulary entry -> dZ column
  const float nw = -w;
#pragma unroll 1
  for (int c = 0; c < kBN / 64; ++c) {
    const int32_t col0 = v0 + c * 64;
    if (col0 + shift >= p.w.dz_cols) break;  // warp-uniform
    // almost every sub-tile of a row lies inside the vocabulary and away from
    // the row's target: there dz = -w e^{z - lse}, the same value the general
    // expression gives (w (0 - p) = (-w) p exactly)
    const bool plain = valid && col0 + 64 <= V && (uint32_t)(y - col0) >= 64u;
    uint4 chunk[8];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      uint32_t raw[32];
      tmem_ld_32x32b_x32(tb + c * 64 + h * 32, raw);
      tmem_ld_wait();
      uint32_t packed[16];
      if (plain) {
#pragma unroll
        for (int k = 0; k < 32; k += 2) {
          const float d0 = nw * ex2_ftz(fmaf(bits_f(raw[k]), kLog2e, -lse_l2));
          const float d1 = nw * ex2_ftz(fmaf(bits_f(raw[k + 1]), kLog2e, -lse_l2));
          packed[k / 2] = pack_bf16x2(d0, d1);
        }
      } else {
#pragma unroll
        for (int k = 0; k < 32; k += 2) {
          float d[2];
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int32_t col = col0 + h * 32 + k + e;
            const float pr = ex2_ftz(fmaf(bits_f(raw[k + e]), kLog2e, -lse_l2));
            const float v = w * ((col == y ? 1.f : 0.f) - pr);
            d[e] = (valid && col < V) ? v : 0.f;
          }
          packed[k / 2] = pack_bf16x2(d[0], d[1]);
        }
      }
#pragma unroll
      for (int q = 0; q < 4; ++q)
        chunk[h * 4 + q] = make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2],
                                      packed[4 * q + 3]);
    }
    const uint32_t sbuf = st.acquire(lane);
    stage_row(sbuf, lane, chunk);
    st.release(lane, sbuf,
               [&](uint32_t a) { tma_store_2d(map_c, a, col0 + shift, (int32_t)(row0 + roff)); });
  }
}

// GEMM_DX: fp32 partial of split s, rows [split * tiles_m * 256 + r] of the
// partial buffer, 32-column sub-tiles through TMA stores in the first
// vocabulary chunk and TMA reduce-adds in the later ones (every element has one
// writer per launch and the chunks run in order, so the sum is deterministic;
// rows >= M hold zeros). Without split-K every dX element has exactly this one
// contribution in the launch, so the lane adds its row's sub-tile straight
// into dX[b, i] (the row the compaction recorded) with 16-byte atomic adds,
// which need no round trip: each element still receives one addition, and the
// split reduction after the last chunk has nothing to do.
__device__ __forceinline__ void dx_sub(const GemmParams& p, const CUtensorMap* map_c,
                                       const Work& wk, float4* drow, int32_t h0, int32_t prow0,
                                       int c, const uint32_t (&raw)[32], int lane, EpiStage& st) {
  if (wk.splits == 1) {  // launch-uniform
    if (drow) {
      // 16-byte pieces of this sub-tile inside the row (H is a multiple of 8)
      const int nq = min(8, ((int32_t)p.g.H - (h0 + c * 32)) / 4);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (q >= nq) break;
        atomicAdd(drow + c * 8 + q, make_float4(bits_f(raw[4 * q]), bits_f(raw[4 * q + 1]),
                                                bits_f(raw[4 * q + 2]), bits_f(raw[4 * q + 3])));
      }
    }
    return;
  }
  uint4 chunk[8];
#pragma unroll
  for (int q = 0; q < 8; ++q)
    chunk[q] = make_uint4(raw[4 * q], raw[4 * q + 1], raw[4 * q + 2], raw[4 * q + 3]);
  const uint32_t sbuf = st.acquire(lane);
  stage_row(sbuf, lane, chunk);
  if (p.chunk == 0)
    st.release(lane, sbuf, [&](uint32_t a) { tma_store_2d(map_c, a, h0 + c * 32, prow0); });
  else
    st.release(lane, sbuf, [&](uint32_t a) { tma_reduce_add_2d(map_c, a, h0 + c * 32, prow0); });
}

// `nb`: the 256-column block of dX this accumulator holds. The TMEM load of
// sub-tile c + 1 is in flight while sub-tile c is written out.
__device__ __forceinline__ void epi_dx(const GemmParams& p, const CUtensorMap* map_c, int32_t M,
                                       const Work& wk, const Unit& t, int32_t nb, int64_t row0,
                                       int lane, uint32_t tb, EpiStage& st) {
  const int32_t h0 = nb * kBN;
  const int32_t nsub = min(kBN / 32, ((int32_t)p.g.H - h0 + 31) / 32);  // inside H
  if (nsub <= 0) return;  // a column block past H (warp-uniform)
  const int32_t prow0 = (int32_t)(t.split * wk.tiles_m * kPairM + row0);
  const int64_t r = row0 + lane;
  float4* drow = nullptr;
  if (wk.splits == 1 && r < M &&
      BGPO_IN_BOUNDS(p.w.err, p.w.rows[r] >= 0 && p.w.rows[r] < p.g.m_cap, KID_DX_GEMM * 16 + 10))
    drow = reinterpret_cast<float4*>(p.dX + (int64_t)p.w.rows[r] * p.g.H + h0);
  uint32_t ra[32], rb[32];
  tmem_ld_32x32b_x32(tb, ra);
  tmem_ld_wait_regs(ra);
#pragma unroll 1
  for (int c = 0; c < nsub; c += 2) {
    if (c + 1 < nsub) tmem_ld_32x32b_x32(tb + (uint32_t)(c + 1) * 32, rb);
    dx_sub(p, map_c, wk, drow, h0, prow0, c, ra, lane, st);
    if (c + 1 < nsub) {
      tmem_ld_wait_regs(rb);
      if (c + 2 < nsub) tmem_ld_32x32b_x32(tb + (uint32_t)(c + 2) * 32, ra);
      dx_sub(p, map_c, wk, drow, h0, prow0, c + 1, rb, lane, st);
      if (c + 2 < nsub) tmem_ld_wait_regs(ra);
    }
  }
}

// GEMM_DW: dW[v, h] += acc through TMA reduce-add of 32 x 32 fp32 sub-tiles
// (the read-modify-write happens at L2; vocabulary rows >= V are clipped).
// Accumulator row r is vocabulary entry v_begin + r.
__device__ __forceinline__ void epi_dw(const GemmParams& p, const CUtensorMap* map_c, const Unit& t,
                                       int64_t row0, int lane, uint32_t tb, EpiStage& st) {
  const int32_t h0 = t.n_blk * kBN;
  const int64_t v = p.v_begin + row0;
  if (v >= p.g.V) return;  // this warp's rows all lie past the vocabulary (warp-uniform)
#pragma unroll 1
  for (int c = 0; c < kBN / 32; ++c) {
    if (h0 + c * 32 >= p.g.H) break;  // warp-uniform
    uint32_t raw[32];
    tmem_ld_32x32b_x32(tb + c * 32, raw);
    tmem_ld_wait();
    uint4 chunk[8];
#pragma unroll
    for (int q = 0; q < 8; ++q)
      chunk[q] = make_uint4(raw[4 * q], raw[4 * q + 1], raw[4 * q + 2], raw[4 * q + 3]);
    const uint32_t sbuf = st.acquire(lane);
    stage_row(sbuf, lane, chunk);
    st.release(lane, sbuf,
               [&](uint32_t a) { tma_reduce_add_2d(map_c, a, h0 + c * 32, (int32_t)v); });
  }
}

template <int KIND>
__device__ __forceinline__ int32_t kernel_id() {
  return KIND == GEMM_FWD ? KID_LMHEAD_FWD
       : KIND == GEMM_DZ  ? KID_LMHEAD_DZ
       : KIND == GEMM_DX  ? KID_DX_GEMM
                          : KID_DW_GEMM;
}

// Sets the abort flag of both CTAs of the pair.
__device__ __forceinline__ void raise_abort(volatile int* abort_flag, uint32_t peer) {
  *abort_flag = 1;
  const uint32_t remote = map_to_cta(smem_addr(const_cast<int*>(abort_flag)), peer);
  asm volatile("st.relaxed.cluster.shared::cluster.u32 [%0], %1;" ::"r"(remote), "r"(1) : "memory");
}

template <int KIND>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    k_gemm(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
           const __grid_constant__ CUtensorMap map_c, const GemmParams p) {
  constexpr int kSt = SmemPlan<KIND>::stages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  constexpr uint32_t kBBytes = Shape<KIND>::b_bytes;
  constexpr int kNacc = Shape<KIND>::nacc;
  constexpr int kBufs = Shape<KIND>::bufs;
  uint8_t* s_a = smem;
  uint8_t* s_b = smem + kSt * kTileABytes;
  uint8_t* s_epi = s_b + kSt * kBBytes;   // 4 warps x 2 staging buffers
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_epi + SmemPlan<KIND>::epi_bytes);
  uint64_t* full = bars;                      // [kSt] TMA (both CTAs) -> MMA; even CTA's
  uint64_t* empty = bars + kSt;           // [kSt] MMA -> TMA of each CTA
  uint64_t* tfull = bars + 2 * kSt;       // [2] MMA -> epilogue of each CTA
  uint64_t* tempty = bars + 2 * kSt + 2;  // [2] epilogues (both CTAs) -> MMA; even CTA's
  uint64_t* done = bars + 2 * kSt + 4;    // MMA drain on abort
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kSt + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* never = reinterpret_cast<volatile int*>(tmem_slot + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();  // 0: even CTA (issues the MMAs), 1: its peer
  const uint32_t peer = rank ^ 1u;
  const int64_t pair = blockIdx.x >> 1;
  const int64_t num_pairs = gridDim.x >> 1;
  int32_t* err = p.w.err;

  int32_t M = 0;
  if (err[ERR_SAMPLE] == p.j) {
    M = err[ERR_M];
  } else if (blockIdx.x == 0 && threadIdx.x == 0) {
    set_device_error(err, kStatusInvalidArg, kernel_id<KIND>() * 16 + 1);
  }
  if (!BGPO_IN_BOUNDS(err, M >= 0 && M <= p.g.m_cap, kernel_id<KIND>() * 16 + 9)) M = 0;
  // first dZ / Xm^T row of this sample: nonzero only when it pairs with a
  // pending sample (the masking set it; the forward does not use dZ)
  const int64_t roff = KIND == GEMM_FWD ? 0 : row_offset(err[ERR_ROW_OFF], p.w.dz_rows, p.g.m_pad);
  // dW: first K row, a multiple of kBK in [0, roff] (see ERR_DW_K0)
  const int64_t k0 = KIND == GEMM_DW ? row_offset(err[ERR_DW_K0], roff + p.g.m_pad, p.g.m_pad) : 0;
  const Work wk = make_work<KIND>(p, M, roff, k0);
  if (KIND == GEMM_DW && blockIdx.x == 0 && threadIdx.x == 0) {
    // a dW GEMM meant to complete a pair whose first sample is not pending
    // adds this sample alone: the other sample's contribution is missing
    if (p.pair_consume && err[ERR_PAIRED] != 1)
      set_device_error(err, kStatusInvalidArg, kernel_id<KIND>() * 16 + 5);
    err[ERR_PEND] = -1;  // nothing waits any more
  }
  // the split reduction after the dX GEMM reads the split count from here
  if (KIND == GEMM_DX && blockIdx.x == 0 && threadIdx.x == 0) err[ERR_DX_SPLITS] = wk.splits;
  if (pair >= wk.units) return;  // both CTAs of the pair, before any allocation

  if (threadIdx.x == 0) {
    for (int s = 0; s < kSt; ++s) {
      mbar_init(smem_addr(&full[s]), 1);    // the even CTA's arrive.expect_tx
      mbar_init(smem_addr(&empty[s]), 1);   // one multicast commit
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_addr(&tfull[a]), 1);
      mbar_init(smem_addr(&tempty[a]), 2 * 4);   // 4 epilogue warps in each CTA
    }
    mbar_init(smem_addr(done), 1);
    *abort_flag = 0;
    *never = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&map_a);
    tma_prefetch_map(&map_b);
    tma_prefetch_map(&map_c);
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_addr(tmem_slot), kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();  // barriers of both CTAs initialised, TMEM allocated
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer (both CTAs) ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      bool issued = false;
      for (int64_t u = pair; u < wk.units && ok; u += num_pairs) {
        const Unit t = unit_of<KIND>(wk, u);
        // the even CTA arms the transaction bytes of both CTAs' copies on its
        // full barrier; the odd CTA's copies only complete_tx on it (a
        // per-stage remote arrive from the odd CTA halved the throughput)
        const uint32_t bytes =
            rank == 0 ? stage_bytes<KIND>(p, t, 0) + stage_bytes<KIND>(p, t, 1) : 0u;
        for (int32_t kb = t.kb0; kb < t.kb0 + t.kb_n; ++kb) {
          if (!mbar_wait(smem_addr(&empty[stage]), phase ^ 1u, abort_flag)) { ok = false; break; }
          const uint32_t cbar = map_to_cta(smem_addr(&full[stage]), 0);
          if (rank == 0) mbar_arrive_expect_tx(smem_addr(&full[stage]), bytes);
          load_stage<KIND>(p, &map_a, &map_b, smem_addr(s_a + stage * kTileABytes),
                           smem_addr(s_b + stage * kBBytes), cbar, t, kb, rank, roff);
          issued = true;
          if (++stage == kSt) { stage = 0; phase ^= 1u; }
        }
      }
      if (!ok) {
        raise_abort(abort_flag, peer);
        set_device_error(err, kStatusTimeout, kernel_id<KIND>() * 16 + 2);
        // let copies already issued land before this CTA can exit
        if (issued) {
          const uint64_t t0 = globaltimer_ns();
          while (globaltimer_ns() - t0 < 2000000ull) {
          }
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer (even CTA) ----------------
    if (rank == 0 && lane == 0) {
      constexpr uint32_t idesc =
          idesc_bf16_f32(kPairM, kBN, Majors<KIND>::a_mn, Majors<KIND>::b_mn);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true, issued = false;
      int it = 0;
      for (int64_t u = pair; u < wk.units && ok; u += num_pairs, ++it) {
        const Unit t = unit_of<KIND>(wk, u);
        const int acc = it % kBufs;
        const uint32_t acc_phase = (uint32_t)(it / kBufs) & 1u;
        if (!mbar_wait(smem_addr(&tempty[acc]), acc_phase ^ 1u, abort_flag)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * kBN);
        for (int32_t kb = 0; kb < t.kb_n; ++kb) {
          if (!mbar_wait(smem_addr(&full[stage]), phase, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sa = smem_addr(s_a + stage * kTileABytes);
          const uint32_t sb = smem_addr(s_b + stage * kBBytes);
#pragma unroll
          for (int k = 0; k < kBK / kUmmaK; ++k) {
            const uint64_t ad = Majors<KIND>::a_mn ? smem_desc_sw128(sa + k * 2048, kMnChunkBytes, 1024)
                                                   : smem_desc_sw128(sa + k * 32, 16, 1024);
#pragma unroll
            for (int g = 0; g < kNacc; ++g) {
              const uint32_t sbg = sb + (uint32_t)g * kTileBBytes;
              const uint64_t bd = Majors<KIND>::b_mn
                                      ? smem_desc_sw128(sbg + k * 2048, kMnChunkBytes, 1024)
                                      : smem_desc_sw128(sbg + k * 32, 16, 1024);
              umma_bf16_pair(d_tmem + (uint32_t)(g * kBN), ad, bd, idesc,
                             (kb > 0 || k > 0) ? 1u : 0u);
            }
          }
          issued = true;
          // frees this stage in both CTAs once these MMAs have read it
          umma_commit_pair(smem_addr(&empty[stage]), kBothCtas);
          if (++stage == kSt) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        umma_commit_pair(smem_addr(&tfull[acc]), kBothCtas);  // accumulators ready
      }
      if (!ok) {
        raise_abort(abort_flag, peer);
        set_device_error(err, kStatusTimeout, kernel_id<KIND>() * 16 + 3);
        if (issued) {
          umma_commit_pair(smem_addr(done), 0x1);
          mbar_wait(smem_addr(done), 0, never);
        }
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue (warps 2..5 of both CTAs) ----------------
    const int quarter = warp & 3;  // TMEM lanes this warp may access: 32*quarter ..
    EpiStage st;
    st.base = smem_addr(s_epi + (uint32_t)(warp - 2) * 2u * kEpiBufBytes);
    st.buf = 0;
    int it = 0;
    bool ok = true;
    for (int64_t u = pair; u < wk.units; u += num_pairs, ++it) {
      const Unit t = unit_of<KIND>(wk, u);
      const int acc = it % kBufs;
      const uint32_t acc_phase = (uint32_t)(it / kBufs) & 1u;
      const bool got = mbar_wait(smem_addr(&tfull[acc]), acc_phase, abort_flag);
      if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
      tc_fence_after();
      const uint32_t tb = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * kBN);
      const int64_t row0 = (int64_t)t.m_blk * kPairM + (int64_t)rank * kBM + quarter * 32;
      if (KIND == GEMM_FWD) epi_fwd(p, &map_c, M, t, row0, lane, tb, st);
      else if (KIND == GEMM_DZ) epi_dz(p, &map_c, M, t, row0, roff, lane, tb, st);
      else if (KIND == GEMM_DX) {
#pragma unroll 1
        for (int g = 0; g < kNacc; ++g)
          epi_dx(p, &map_c, M, wk, t, t.n_blk * kNacc + g, row0, lane, tb + (uint32_t)(g * kBN), st);
      }
      else epi_dw(p, &map_c, t, row0, lane, tb, st);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(map_to_cta(smem_addr(&tempty[acc]), 0));
    }
    // every bulk store / reduction of this warp has completed before exit
    if (lane == 0) bulk_wait_group<0>();
    __syncwarp();
    if (!ok) {
      raise_abort(abort_flag, peer);
      if (lane == 0) set_device_error(err, kStatusTimeout, kernel_id<KIND>() * 16 + 4);
    }
  }

  tc_fence_before();
  cluster_sync();  // no CTA of the pair still reads the other's shared memory
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
}

template <int KIND>
cudaError_t launch_kind(const CUtensorMap& ma, const CUtensorMap& mb, const CUtensorMap& mc,
                        const GemmParams& p, cudaStream_t s) {
  constexpr uint32_t smem = SmemPlan<KIND>::bytes;
  cudaError_t e = cudaFuncSetAttribute(k_gemm<KIND>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  k_gemm<KIND><<<2 * p.num_pairs, kThreads, smem, s>>>(ma, mb, mc, p);
  return cudaGetLastError();
}

}  // namespace

int gemm_num_pairs(int num_sms) {
  static int cached = 0;
  static std::once_flag once;
  std::call_once(once, [num_sms] {
    int clusters = 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)num_sms, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = SmemPlan<GEMM_DX>::bytes;
    if (cudaFuncSetAttribute(k_gemm<GEMM_DX>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)SmemPlan<GEMM_DX>::bytes) == cudaSuccess &&
        cudaOccupancyMaxActiveClusters(&clusters, k_gemm<GEMM_DX>, &cfg) == cudaSuccess &&
        clusters > 0)
      cached = clusters;
    else
      cudaGetLastError();
  });
  const int half = num_sms / 2;
  return (cached > 0 && cached < half) ? cached : half;
}

cudaError_t launch_gemm(GemmKind kind, const CUtensorMap& map_a, const CUtensorMap& map_b,
                        const CUtensorMap& map_c, const GemmArgs& a, const WsPtrs& w,
                        cudaStream_t s) {
  GemmParams p;
  p.g = a.g;
  p.num_pairs = a.num_pairs;
  p.j = a.j;
  p.v_begin = a.v_begin;
  p.v_end = a.v_end;
  p.dz_col0 = a.dz_col0;
  p.chunk = a.chunk;
  p.w = w;
  p.coef = a.coef;
  p.dW = a.dW;
  p.dX = a.dX;
  p.pair_consume = a.pair_consume;
  switch (kind) {
    case GEMM_FWD: return launch_kind<GEMM_FWD>(map_a, map_b, map_c, p, s);
    case GEMM_DZ: return launch_kind<GEMM_DZ>(map_a, map_b, map_c, p, s);
    case GEMM_DX: return launch_kind<GEMM_DX>(map_a, map_b, map_c, p, s);
    case GEMM_DW: return launch_kind<GEMM_DW>(map_a, map_b, map_c, p, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace bgpo

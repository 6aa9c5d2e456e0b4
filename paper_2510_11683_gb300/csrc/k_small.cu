// Non-GEMM kernels of the BGPO LM-head ELBO path: the forward masking process
// with row compaction, the gather of masked hidden states, the log-sum-exp
// combine, the per-sequence ELBO reduction (Eq. 4), the bound coefficients
// (Eq. 10, 13), dL/dz from the logits the forward kept, the split-K reduction
// of dX, the transpose of the gathered rows for the dW GEMM and the group
// advantages (Eq. 18).
#include <math.h>

#include "bgpo_device.cuh"
#include "bgpo_internal.h"
#include "philox.cuh"

namespace bgpo {

namespace {

constexpr int32_t kStatusInvalidArg = 1;   // BGPO_ERR_INVALID_ARG
constexpr int32_t kStatusNonfinite = 5;    // BGPO_ERR_NONFINITE
constexpr float kLog2e = 1.4426950408889634f;

// Masked rows of the sample the workspace holds, or 0 (and an error) when the
// workspace holds another sample than `j`.
__device__ __forceinline__ int32_t rows_of_sample(int32_t* err, int32_t j, int32_t kid) {
  const int32_t tag = err[ERR_SAMPLE];
  if (tag != j) {
    if (blockIdx.x == 0 && threadIdx.x == 0) set_device_error(err, kStatusInvalidArg, kid * 16 + 1);
    return 0;
  }
  return err[ERR_M];
}

// ---------------------------------------------------------------------------
// Forward masking process (Sec. 2.1; Eq. 3, 5) + stable compaction.
// One CTA of 1024 threads first draws every sequence's t (one Philox block
// each, kept in the workspace), then walks the (b, q) mask blocks in ascending
// order, 1024 blocks per round; a block-wide exclusive scan places every
// masked position (b, i) at its rank, so rows[] is sorted by b * R + i.
// ---------------------------------------------------------------------------
constexpr int kScanThreads = 1024;

__global__ void __launch_bounds__(kScanThreads) k_mask_compact(MaskArgs a, WsPtrs w) {
  __shared__ int32_t warp_excl[32];
  __shared__ int32_t s_carry;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int64_t Q = ((int64_t)a.R + 3) / 4;
  const int64_t nblk = (int64_t)a.B * Q;
  const uint64_t d_over_2_24 = (a.t_mode == 1) ? (uint64_t)a.n_t : 1ull;   // D / 2^24
  if (tid == 0) s_carry = 0;
  // t of every sequence: T = u24 + 1 (i.i.d.) or j 2^24 + u24 + 1 (stratified)
  for (int32_t b = tid; b < a.B; b += kScanThreads) {
    const uint64_t bg = (uint64_t)b + (uint64_t)a.b_offset;   // global sequence index
    const PhiloxOut ot = philox4x64_10(0, bg, (uint64_t)a.j, kStreamT, a.seed, 0);
    const uint64_t u = ot.w[0] >> kU24Shift;
    const uint64_t T = (a.t_mode == 1) ? ((uint64_t)a.j << 24) + u + 1 : u + 1;
    const float tf = (float)((double)T / (double)(d_over_2_24 << 24));
    w.t[b] = tf;
    w.tnum[2 * b] = (uint32_t)T;
    w.tnum[2 * b + 1] = (uint32_t)(T >> 32);
    if (a.t_out) a.t_out[b] = tf;
  }
  __syncthreads();  // the block's T values are visible to every thread
  for (int64_t base = 0; base < nblk; base += kScanThreads) {
    const int64_t e = base + tid;
    int32_t cnt = 0;
    uint32_t bits = 0;
    int32_t b = 0, q = 0;
    if (e < nblk) {
      b = (int32_t)(e / Q);
      q = (int32_t)(e % Q);
      const uint64_t bg = (uint64_t)b + (uint64_t)a.b_offset;   // global sequence index
      const int32_t len = a.resp_len ? min(max(a.resp_len[b], 0), a.R) : a.R;
      const uint64_t T = (uint64_t)w.tnum[2 * b] | ((uint64_t)w.tnum[2 * b + 1] << 32);
      const PhiloxOut om = philox4x64_10((uint64_t)q, bg, (uint64_t)a.j, kStreamMask, a.seed, 0);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int32_t i = 4 * q + k;
        if (i < a.R) {
          // u24 / 2^24 < T / D  <=>  u24 * (D / 2^24) < T   (exact integers);
          // padding positions (i >= len) are never masked
          const uint32_t bit = (i < len && (om.w[k] >> kU24Shift) * d_over_2_24 < T) ? 1u : 0u;
          bits |= bit << k;
          cnt += (int32_t)bit;
          if (a.mask_out) a.mask_out[(int64_t)b * a.R + i] = (uint8_t)bit;
        }
      }
    }
    // block-wide exclusive scan of cnt
    int32_t incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    if (lane == 31) warp_excl[wid] = incl;
    __syncthreads();
    if (wid == 0) {
      const int32_t v = warp_excl[lane];
      int32_t vi = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int32_t n = __shfl_up_sync(0xffffffffu, vi, o);
        if (lane >= o) vi += n;
      }
      warp_excl[lane] = vi - v;
    }
    __syncthreads();
    const int32_t excl = s_carry + warp_excl[wid] + incl - cnt;
    if (e < nblk) {
      if (q == 0) w.seg_off[b] = excl;
      int32_t pos = excl;
#pragma unroll
      for (int k = 0; k < 4; ++k)
        if ((bits >> k) & 1u) {
          if (BGPO_IN_BOUNDS(w.err, pos < a.B * a.R, KID_MASK_COMPACT * 16 + 9))
            w.rows[pos] = b * a.R + 4 * q + k;
          ++pos;
        }
    }
    __syncthreads();
    if (tid == kScanThreads - 1) s_carry = excl + cnt;
    __syncthreads();
  }
  if (tid == 0) {
    const int32_t M = s_carry;
    w.seg_off[a.B] = M;
    // dW pairing: an odd sample pairs with sample j - 1 when that sample's
    // backward left its rows pending in this workspace and no other sample has
    // been masked here since (masking sample j again keeps the pairing). A
    // pending sample that no pairing takes up would lose its dW contribution:
    // that is an error, unless the pending sample itself is masked again (its
    // backward will then run again).
    const int32_t prev = w.err[ERR_SAMPLE];
    const int32_t pend = w.err[ERR_PEND];
    const bool pending = (pend & (int32_t)0xFFFF0000u) == pend_tag(0);
    const int32_t pj = pend & 0xFFFF;
    const bool paired = a.pair_dw && (a.j & 1) && pending && pj == a.j - 1 &&
                        (prev == a.j - 1 || prev == a.j);
    if (paired) {
      w.err[ERR_ROW_OFF] = w.err[ERR_PEND_OFF];
      w.err[ERR_PAIRED] = 1;
    } else {
      if (pending && pj != a.j) set_device_error(w.err, kStatusInvalidArg, KID_MASK_COMPACT * 16 + 5);
      w.err[ERR_ROW_OFF] = 0;
      w.err[ERR_PAIRED] = 0;
      w.err[ERR_PEND] = -1;
    }
    w.err[ERR_M] = M;
    w.err[ERR_SAMPLE] = a.j;
    w.err[ERR_LOGITS] = 0;  // no forward of this sample has kept its logits yet
  }
}

// ---------------------------------------------------------------------------
// Gather of the masked rows' hidden states (the indicator of Eq. 4 selects
// them): Xm[r] = X[b, P + i] with 16-byte vector copies, one warp per row.
// Rows [M, round_up(M, 256)) are zero-filled so that the GEMM pair tiles and
// the K padding of the dW GEMM read zeros.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_gather(Geometry g, int32_t j, const uint4* __restrict__ X,
                                                const int32_t* __restrict__ Y, WsPtrs w) {
  const int32_t M = rows_of_sample(w.err, j, KID_GATHER);
  if (!BGPO_IN_BOUNDS(w.err, M <= g.m_cap, KID_GATHER * 16 + 9)) return;
  const int64_t r = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= round_up(M, kPairM)) return;
  const int64_t nvec = g.H / 8;
  uint4* dst = reinterpret_cast<uint4*>(w.xm) + r * nvec;
  if (r < M) {
    const int32_t idx = w.rows[r];
    if (!BGPO_IN_BOUNDS(w.err, idx >= 0 && idx < g.m_cap, KID_GATHER * 16 + 10)) return;
    const int64_t b = idx / g.R, i = idx % g.R;
    const uint4* src = X + (b * (g.P + g.R) + g.P + i) * nvec;
    // 8 loads of 16 bytes in flight per lane before their stores
    for (int64_t v0 = lane; v0 < nvec; v0 += 32 * 8) {
      uint4 q[8];
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if (v0 + 32 * k < nvec) q[k] = __ldg(src + v0 + 32 * k);
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if (v0 + 32 * k < nvec) dst[v0 + 32 * k] = q[k];
    }
    if (lane == 0) {
      const int32_t y = __ldg(Y + idx);
      (void)BGPO_IN_BOUNDS(w.err, y >= 0 && y < g.V, KID_GATHER * 16 + 11);  // a target outside V
      w.tgt[r] = y;
    }
  } else {
    const uint4 z = make_uint4(0, 0, 0, 0);
    for (int64_t v = lane; v < nvec; v += 32) dst[v] = z;
    if (lane == 0) w.tgt[r] = 0;
  }
}

// (m, s) pairs represent s * e^m; merging keeps the larger exponent.
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) { m = m2; s = s2; return; }
  if (m2 > m) { s = s * expf(m - m2) + s2; m = m2; }
  else        { s = s + s2 * expf(m2 - m); }
}

constexpr int kLseBatch = 8;

// ---------------------------------------------------------------------------
// log-sum-exp of each masked row from the per-vocab-tile partials, then
// log p(y_r) = z_{r, y_r} - lse_r. One warp per row, fixed merge order.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_lse_combine(Geometry g, int32_t j, bool kept_logits,
                                                     WsPtrs w) {
  const int32_t M = rows_of_sample(w.err, j, KID_LSE_COMBINE);
  if (blockIdx.x == 0 && threadIdx.x == 0)
    w.err[ERR_LOGITS] = (kept_logits && w.err[ERR_SAMPLE] == j) ? 1 : 0;
  const int64_t r = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= M) return;
  float m = -INFINITY, s = 0.f;
  const float2* part = w.part + r * g.n_vt;
  // each lane merges partials lane, lane + 32, ... in order; kLseBatch loads
  // are in flight before the merges that need them
  for (int64_t i = lane; i < g.n_vt; i += 32 * kLseBatch) {
    float2 q[kLseBatch];
#pragma unroll
    for (int k = 0; k < kLseBatch; ++k) {
      const int64_t idx = i + 32 * k;
      q[k] = idx < g.n_vt ? part[idx] : make_float2(-INFINITY, 0.f);
    }
#pragma unroll
    for (int k = 0; k < kLseBatch; ++k) lse_merge(m, s, q[k].x, q[k].y);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    lse_merge(m, s, m2, s2);
  }
  if (lane == 0) {
    const float lse = m + logf(s);
    w.lse[r] = lse;
    w.logp[r] = w.tgt_logit[r] - lse;
  }
}

// ---------------------------------------------------------------------------
// dL/dz of the masked rows, one vocabulary chunk [v0, v1) of the backward, from
// the logits the forward kept:
//   dz_{r,v} = w_r (1[v = y_r] - e^{z_{r,v} - lse_r}),  w_r = coef_b / t_b
// (gradient of Eq. 4 weighted by dL/dl), bf16, zero for rows in
// [M, round_up(M, 256)) and columns at or past V: the arithmetic of the
// GEMM_DZ epilogue on the same fp32 logits, so both give identical bits.
// Entry v lands in dZ column v - v0 (a chunk-local buffer) or v (a
// whole-vocabulary one). HBM-bound: each row streams 4 bytes in and 2 bytes out
// per column. Work items are (row, 8192-column piece); each thread has kDzVec
// independent 32-byte loads in flight before it computes.
// When the workspace holds no logits of sample j the kernel records
// BGPO_ERR_INVALID_ARG and invalidates the sample tag, so that the dX / dW
// kernels after it do no work.
// ---------------------------------------------------------------------------
constexpr int kDzThreads = 256;
constexpr int kDzVec = 4;                           // 8-column vectors per thread per item
constexpr int kDzItemVecs = kDzThreads * kDzVec;    // 1024 vectors = 8192 columns

__global__ void __launch_bounds__(kDzThreads, 4)
    k_dz_from_logits(Geometry g, int32_t j, int64_t chunk, const float* __restrict__ coef,
                     WsPtrs w) {
  const int32_t M = rows_of_sample(w.err, j, KID_DZ_FROM_LOGITS);
  if (w.err[ERR_LOGITS] != 1) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      set_device_error(w.err, kStatusInvalidArg, KID_DZ_FROM_LOGITS * 16 + 2);
      w.err[ERR_SAMPLE] = -1;
    }
    return;
  }
  if (!BGPO_IN_BOUNDS(w.err, M <= g.m_cap, KID_DZ_FROM_LOGITS * 16 + 9)) return;
  const int64_t v_begin = chunk_begin(g, chunk);
  // 8-column vectors of the chunk (its width rounded up to 64 columns), of a
  // kept-logit row and of a dZ row
  const int64_t nvec = round_up(chunk_end(g, chunk) - v_begin, 64) / 8;
  const int64_t zvec = g.v_pad / 8;
  const int64_t dvec = w.dz_cols / 8;
  const int64_t per_row = ceil_div(nvec, kDzItemVecs);
  const int64_t items = round_up(M, kPairM) * per_row;
  const float4* __restrict__ zc = reinterpret_cast<const float4*>(w.zc) + v_begin / 4;
  // this sample's dZ rows start at the pairing offset (0 without pairing)
  uint4* __restrict__ dz = reinterpret_cast<uint4*>(w.dz) +
                           row_offset(w.err[ERR_ROW_OFF], w.dz_rows, g.m_pad) * dvec +
                           (w.dz_chunk_local ? 0 : v_begin / 8);
  const int32_t V = (int32_t)g.V;
  for (int64_t q = blockIdx.x; q < items; q += gridDim.x) {
    const int64_t r = q / per_row;
    const int64_t v0 = (q % per_row) * kDzItemVecs + threadIdx.x;
    const bool valid = r < M;
    float wr = 0.f, lse_l2 = 0.f;
    int32_t y = -1;
    if (valid) {
      const int32_t idx = w.rows[r];
      if (!BGPO_IN_BOUNDS(w.err, idx >= 0 && idx < g.m_cap, KID_DZ_FROM_LOGITS * 16 + 10)) continue;
      const int32_t b = idx / (int32_t)g.R;
      wr = coef[b] / w.t[b];
      lse_l2 = w.lse[r] * kLog2e;
      y = w.tgt[r];
    }
    float4 z[kDzVec][2];
#pragma unroll
    for (int k = 0; k < kDzVec; ++k) {
      const int64_t v = v0 + k * kDzThreads;
      if (valid && v < nvec) {
        const float4* src = zc + r * zvec * 2 + v * 2;
        z[k][0] = __ldcs(src);
        z[k][1] = __ldcs(src + 1);
      } else {
        z[k][0] = z[k][1] = make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
#pragma unroll
    for (int k = 0; k < kDzVec; ++k) {
      const int64_t v = v0 + k * kDzThreads;
      if (v >= nvec) continue;
      const float zz[8] = {z[k][0].x, z[k][0].y, z[k][0].z, z[k][0].w,
                           z[k][1].x, z[k][1].y, z[k][1].z, z[k][1].w};
      uint32_t packed[4];
#pragma unroll
      for (int e = 0; e < 8; e += 2) {
        float d[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int32_t col = (int32_t)(v_begin + v * 8) + e + h;
          const float pr = ex2_ftz(fmaf(zz[e + h], kLog2e, -lse_l2));
          const float val = wr * ((col == y ? 1.f : 0.f) - pr);
          d[h] = (valid && col < V) ? val : 0.f;
        }
        const __nv_bfloat162 hv = __floats2bfloat162_rn(d[0], d[1]);
        packed[e / 2] = *reinterpret_cast<const uint32_t*>(&hv);
      }
      dz[r * dvec + v] = make_uint4(packed[0], packed[1], packed[2], packed[3]);
    }
  }
}

// ---------------------------------------------------------------------------
// Eq. 4: l_b = (1/t_b) * sum over sequence b's masked rows of log p. One warp
// per sequence, lane-strided sums then a fixed xor tree (deterministic).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_seq_reduce(Geometry g, int32_t j, WsPtrs w, float* ell_out) {
  const int32_t M = rows_of_sample(w.err, j, KID_SEQ_REDUCE);
  const int64_t b = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (b >= g.B) return;
  float acc = 0.f;
  if (M > 0) {
    const int32_t lo = w.seg_off[b], hi = w.seg_off[b + 1];
    if (BGPO_IN_BOUNDS(w.err, 0 <= lo && lo <= hi && hi <= M && M <= g.m_cap, KID_SEQ_REDUCE * 16 + 9))
      for (int32_t r = lo + lane; r < hi; r += 32) acc += w.logp[r];
  }
  acc = warp_sum(acc);
  if (lane == 0) ell_out[b] = acc / w.t[b];
}

// ---------------------------------------------------------------------------
// Eq. 10 and 13 (Algorithm 1: L_j = -loss_scale * g_j):
//   d = l - l_old; A >= 0: g = (1 + d) A / n_t, dg/dl = A / n_t (Lemma 1)
//                  A <  0: g = e^d A / n_t,    dg/dl = e^d A / n_t (Lemma 2)
// ---------------------------------------------------------------------------
__global__ void k_bound_coeffs(int32_t B, int32_t n_t, float loss_scale, const float* __restrict__ ell,
                               const float* __restrict__ ell_old, const float* __restrict__ A,
                               float* coef_out, float* g_out, int32_t* err) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const float d = ell[b] - ell_old[b];
  const float a = A[b];
  const bool taylor = a >= 0.f;
  const float kappa = taylor ? 1.f : expf(d);
  const float inv_nt = 1.f / (float)n_t;
  const float g = taylor ? (1.f + d) * a * inv_nt : kappa * a * inv_nt;
  const float coef = -loss_scale * a * kappa * inv_nt;
  coef_out[b] = coef;
  if (g_out) g_out[b] = g;
  if (!isfinite(g) || !isfinite(coef)) set_device_error(err, kStatusNonfinite, KID_BOUND_COEFFS * 16);
}

// ---------------------------------------------------------------------------
// VRPO (Eq. 7): R_hat = e^{mean_j (l - l_old)} A and dL/dl_{b,j} =
// -loss_scale A e^{mean_j d} / n_t for every j (Sec. 3.2). l, l_old [n_t, B].
// ---------------------------------------------------------------------------
__global__ void k_vrpo_coeffs(int32_t B, int32_t n_t, float loss_scale, const float* __restrict__ ell,
                              const float* __restrict__ ell_old, const float* __restrict__ A,
                              float* coef_out, float* R_out, int32_t* err) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  float sum_d = 0.f;
  for (int j = 0; j < n_t; ++j) sum_d += ell[(int64_t)j * B + b] - ell_old[(int64_t)j * B + b];
  const float inv_nt = 1.f / (float)n_t;
  const float e = expf(sum_d * inv_nt);
  const float a = A[b];
  const float R = e * a;
  const float coef = -loss_scale * a * e * inv_nt;
  coef_out[b] = coef;
  if (R_out) R_out[b] = R;
  if (!isfinite(R) || !isfinite(coef)) set_device_error(err, kStatusNonfinite, KID_VRPO_COEFFS * 16);
}

// ---------------------------------------------------------------------------
// dX[b, i, :] += sum_s partial_s[r, :] over the split-K partials of the dX GEMM
// (fixed split order; rows are unique within a sample, so no atomics). With a
// single split the GEMM's epilogue has already added its tile into dX. Each
// thread keeps kDxrVec 16-byte loads of a split (and of the dX row) in flight
// at once.
// ---------------------------------------------------------------------------
constexpr int kDxrThreads = 256;
constexpr int kDxrVec = 4;

__global__ void __launch_bounds__(kDxrThreads) k_dx_reduce(Geometry g, int32_t j, WsPtrs w,
                                                           float* __restrict__ dX) {
  const int32_t M = rows_of_sample(w.err, j, KID_DX_REDUCE);
  const int64_t r = blockIdx.x;
  if (r >= M) return;
  const int64_t mb = ceil_div(M, kPairM);
  const int S = w.err[ERR_DX_SPLITS];  // written by the dX GEMM of this sample
  if (S == 1) return;
  if (S < 1 || S > kMaxSplits || S * mb > dxp_row_block_cap(g)) {  // not a count it can write
    if (r == 0 && threadIdx.x == 0) set_device_error(w.err, kStatusInvalidArg, KID_DX_REDUCE * 16 + 2);
    return;
  }
  const int64_t split_stride = mb * kPairM * g.H / 4;
  const int32_t idx = w.rows[r];
  if (!BGPO_IN_BOUNDS(w.err, idx >= 0 && idx < g.m_cap, KID_DX_REDUCE * 16 + 9)) return;
  const float4* __restrict__ src = reinterpret_cast<const float4*>(w.dxp) + r * (g.H / 4);
  float4* dst = reinterpret_cast<float4*>(dX) + (int64_t)idx * (g.H / 4);
  const int64_t nvec = g.H / 4;
  for (int64_t h0 = threadIdx.x; h0 < nvec; h0 += (int64_t)kDxrThreads * kDxrVec) {
    float4 acc[kDxrVec], o[kDxrVec];
#pragma unroll
    for (int k = 0; k < kDxrVec; ++k) {
      const int64_t h = h0 + (int64_t)k * kDxrThreads;
      const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
      acc[k] = h < nvec ? src[h] : z;
      o[k] = h < nvec ? dst[h] : z;
    }
    for (int s = 1; s < S; ++s) {
      float4 v[kDxrVec];
#pragma unroll
      for (int k = 0; k < kDxrVec; ++k) {
        const int64_t h = h0 + (int64_t)k * kDxrThreads;
        v[k] = h < nvec ? src[s * split_stride + h] : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int k = 0; k < kDxrVec; ++k) {
        acc[k].x += v[k].x; acc[k].y += v[k].y; acc[k].z += v[k].z; acc[k].w += v[k].w;
      }
    }
#pragma unroll
    for (int k = 0; k < kDxrVec; ++k) {
      const int64_t h = h0 + (int64_t)k * kDxrThreads;
      if (h < nvec) {
        o[k].x += acc[k].x; o[k].y += acc[k].y; o[k].z += acc[k].z; o[k].w += acc[k].w;
        dst[h] = o[k];
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Xm^T [H, dz_rows] from Xm [m_pad, H] for rows [0, round_up(M, 256)) of the
// current sample, into columns [off, off + round_up(M, 256)) with off the
// pairing offset (0 without pairing; rows past M are the gather's zeros, so the
// K padding of the dW GEMM reads zeros). With Xm^T the dW GEMM's B operand is
// K-major: one K-major and two MN-major boxes per stage instead of four
// MN-major boxes, which measured 12% faster. A block moves a 256-row x
// 64-column tile through shared memory with 16-byte global loads and stores,
// all 8 of a thread's loads in flight at once; the row pitch of 66 elements
// keeps the column reads to two-way bank conflicts.
// ---------------------------------------------------------------------------
constexpr int kTrRows = kPairM;   // one pair tile of rows per block
constexpr int kTrCols = 64;
constexpr int kTrPitch = kTrCols + 2;
constexpr int kTrThreads = 256;
constexpr int kTrChunks = kTrRows * kTrCols / 8 / kTrThreads;   // 16-byte chunks per thread

__global__ void __launch_bounds__(kTrThreads) k_xm_transpose(Geometry g, int32_t j, bool defer,
                                                             WsPtrs w) {
  const int32_t M = rows_of_sample(w.err, j, KID_XM_TRANSPOSE);
  if (!BGPO_IN_BOUNDS(w.err, M <= g.m_cap, KID_XM_TRANSPOSE * 16 + 9)) return;
  const int64_t off = row_offset(w.err[ERR_ROW_OFF], w.dz_rows, g.m_pad);
  if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) {
    // the dW GEMM after this kernel adds the pending partner's rows [0, off)
    // only while the partner is still pending (a repeated backward of this
    // sample adds its own rows alone)
    w.err[ERR_DW_K0] = (j > 0 && w.err[ERR_PEND] == pend_tag(j - 1)) ? 0 : (int32_t)off;
    if (defer) {
      // the next sample's rows follow this sample's, from the next K block on
      w.err[ERR_PEND_OFF] = (int32_t)round_up(M, kBK);
      w.err[ERR_PEND] = pend_tag(j);
    }
  }
  const int64_t r0 = (int64_t)blockIdx.x * kTrRows;
  const int64_t h0 = (int64_t)blockIdx.y * kTrCols;
  if (r0 >= round_up(M, kPairM)) return;  // block-uniform
  __shared__ __align__(16) uint16_t tile[kTrRows * kTrPitch];
  const uint16_t* __restrict__ xm = static_cast<const uint16_t*>(w.xm);
  uint16_t* __restrict__ xmT = static_cast<uint16_t*>(w.xmT);
  uint4 v[kTrChunks];
#pragma unroll
  for (int i = 0; i < kTrChunks; ++i) {   // chunk c: row c / 8, columns (c % 8) * 8 ..
    const int c = threadIdx.x + i * kTrThreads;
    // H is a multiple of 8: a chunk lies wholly inside or wholly past the row
    v[i] = h0 + (c % 8) * 8 < g.H
               ? *reinterpret_cast<const uint4*>(xm + (r0 + c / 8) * g.H + h0 + (c % 8) * 8)
               : make_uint4(0, 0, 0, 0);
  }
#pragma unroll
  for (int i = 0; i < kTrChunks; ++i) {
    const int c = threadIdx.x + i * kTrThreads;
    uint32_t* dst = reinterpret_cast<uint32_t*>(tile + (c / 8) * kTrPitch + (c % 8) * 8);
    dst[0] = v[i].x; dst[1] = v[i].y; dst[2] = v[i].z; dst[3] = v[i].w;
  }
  __syncthreads();
#pragma unroll
  for (int i = 0; i < kTrChunks; ++i) {
    // output chunk c: column hh of the tile, 8 rows from rr; 8 consecutive
    // threads write one 128-byte segment of an Xm^T row
    const int c = threadIdx.x + i * kTrThreads;
    const int hh = (c / 8) % kTrCols;
    const int rr = (c / (8 * kTrCols)) * 64 + (c % 8) * 8;
    if (h0 + hh >= g.H) continue;     // Xm^T has H rows
    uint32_t word[4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
      word[k] = (uint32_t)tile[(rr + 2 * k) * kTrPitch + hh] |
                ((uint32_t)tile[(rr + 2 * k + 1) * kTrPitch + hh] << 16);
    *reinterpret_cast<uint4*>(xmT + (h0 + hh) * w.dz_rows + off + r0 + rr) =
        make_uint4(word[0], word[1], word[2], word[3]);
  }
}

// ---------------------------------------------------------------------------
// Eq. 18 over consecutive groups of G rewards (population std; 0 if std = 0).
// ---------------------------------------------------------------------------
__global__ void k_group_advantage(int32_t B, int32_t G, const float* __restrict__ r, float* A) {
  const int64_t grp = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (grp * G >= B) return;
  const float* x = r + grp * G;
  float mean = 0.f;
  for (int k = 0; k < G; ++k) mean += x[k];
  mean /= (float)G;
  float var = 0.f;
  for (int k = 0; k < G; ++k) var += (x[k] - mean) * (x[k] - mean);
  const float sd = sqrtf(var / (float)G);
  for (int k = 0; k < G; ++k) A[grp * G + k] = sd > 0.f ? (x[k] - mean) / sd : 0.f;
}

// ---------------------------------------------------------------------------
// Self-test of the bounded waits every kernel here uses: one warp waits on an
// mbarrier that nothing arrives at; the wait must give up after timeout_ns and
// record BGPO_ERR_TIMEOUT in the error word.
// ---------------------------------------------------------------------------
__global__ void k_selftest_wait(int32_t* err, uint64_t timeout_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  const uint32_t b = smem_addr(&bar);
  if (threadIdx.x == 0) {
    mbar_init(b, 1);
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncwarp();
  const bool done = mbar_wait_timeout(b, 0, &abort_flag, timeout_ns);
  if (!__all_sync(0xffffffffu, done) && threadIdx.x == 0)
    set_device_error(err, 8 /* BGPO_ERR_TIMEOUT */, KID_SELFTEST_WAIT * 16);
}

}  // namespace

cudaError_t launch_selftest_wait(int32_t* err, uint64_t timeout_ns, cudaStream_t s) {
  k_selftest_wait<<<1, 32, 0, s>>>(err, timeout_ns);
  return cudaGetLastError();
}

WsPtrs ws_pointers(void* ws, const WsLayout& L, bool forward_only) {
  char* base = static_cast<char*>(ws);
  WsPtrs p;
  p.err = reinterpret_cast<int32_t*>(base + L.err);
  p.t = reinterpret_cast<float*>(base + L.t);
  p.tnum = reinterpret_cast<uint32_t*>(base + L.tnum);
  p.seg_off = reinterpret_cast<int32_t*>(base + L.seg_off);
  p.rows = reinterpret_cast<int32_t*>(base + L.rows);
  p.tgt = reinterpret_cast<int32_t*>(base + L.tgt);
  p.tgt_logit = reinterpret_cast<float*>(base + L.tgt_logit);
  p.lse = reinterpret_cast<float*>(base + L.lse);
  p.logp = reinterpret_cast<float*>(base + L.logp);
  p.part = reinterpret_cast<float2*>(base + L.part);
  p.xm = base + L.xm;
  p.xmT = forward_only ? nullptr : base + L.xmT;
  p.dz = forward_only ? nullptr : base + L.dz;
  p.dz_rows = forward_only ? 0 : (int64_t)L.dz_rows;
  p.dz_cols = forward_only ? 0 : (int64_t)L.dz_cols;
  p.dz_chunk_local = !forward_only && L.dz_chunk_local;
  p.dxp = forward_only ? nullptr : reinterpret_cast<float*>(base + L.dxp);
  p.zc = (!forward_only && L.zc_bytes) ? reinterpret_cast<float*>(base + L.zc) : nullptr;
  return p;
}

cudaError_t launch_mask_compact(const MaskArgs& a, const WsPtrs& w, cudaStream_t s) {
  k_mask_compact<<<1, kScanThreads, 0, s>>>(a, w);
  return cudaGetLastError();
}

cudaError_t launch_gather(const Geometry& g, int32_t j, const void* X, const int32_t* Y,
                          const WsPtrs& w, cudaStream_t s) {
  const unsigned grid = (unsigned)ceil_div(g.m_pad, 8);
  k_gather<<<grid, 256, 0, s>>>(g, j, static_cast<const uint4*>(X), Y, w);
  return cudaGetLastError();
}

cudaError_t launch_lse_combine(const Geometry& g, int32_t j, bool kept_logits, const WsPtrs& w,
                               cudaStream_t s) {
  const unsigned grid = (unsigned)ceil_div(g.m_cap, 8);
  k_lse_combine<<<grid, 256, 0, s>>>(g, j, kept_logits, w);
  return cudaGetLastError();
}

cudaError_t launch_dz_from_logits(const Geometry& g, int32_t j, int64_t chunk, const float* coef,
                                  int num_sms, const WsPtrs& w, cudaStream_t s) {
  // 4 resident CTAs per SM; never more CTAs than the largest sample has items
  const int64_t most = g.m_pad * ceil_div(g.vc / 8, kDzItemVecs);
  const int64_t grid = most < 4 * (int64_t)num_sms ? most : 4 * (int64_t)num_sms;
  k_dz_from_logits<<<(unsigned)grid, kDzThreads, 0, s>>>(g, j, chunk, coef, w);
  return cudaGetLastError();
}

cudaError_t launch_seq_reduce(const Geometry& g, int32_t j, const WsPtrs& w, float* ell_out,
                              cudaStream_t s) {
  const unsigned grid = (unsigned)ceil_div(g.B, 8);
  k_seq_reduce<<<grid, 256, 0, s>>>(g, j, w, ell_out);
  return cudaGetLastError();
}

cudaError_t launch_bound_coeffs(int32_t B, int32_t n_t, float loss_scale, const float* ell,
                                const float* ell_old, const float* A, float* coef_out,
                                float* g_out, const WsPtrs& w, cudaStream_t s) {
  k_bound_coeffs<<<(unsigned)ceil_div(B, 256), 256, 0, s>>>(B, n_t, loss_scale, ell, ell_old, A,
                                                            coef_out, g_out, w.err);
  return cudaGetLastError();
}

cudaError_t launch_vrpo_coeffs(int32_t B, int32_t n_t, float loss_scale, const float* ell,
                               const float* ell_old, const float* A, float* coef_out, float* R_out,
                               const WsPtrs& w, cudaStream_t s) {
  k_vrpo_coeffs<<<(unsigned)ceil_div(B, 256), 256, 0, s>>>(B, n_t, loss_scale, ell, ell_old, A,
                                                           coef_out, R_out, w.err);
  return cudaGetLastError();
}

cudaError_t launch_dx_reduce(const Geometry& g, int32_t j, const WsPtrs& w, float* dX,
                             cudaStream_t s) {
  k_dx_reduce<<<(unsigned)g.m_cap, kDxrThreads, 0, s>>>(g, j, w, dX);
  return cudaGetLastError();
}

cudaError_t launch_xm_transpose(const Geometry& g, int32_t j, bool defer, const WsPtrs& w,
                                cudaStream_t s) {
  const dim3 grid((unsigned)(g.m_pad / kTrRows), (unsigned)ceil_div(g.H, kTrCols));
  k_xm_transpose<<<grid, kTrThreads, 0, s>>>(g, j, defer, w);
  return cudaGetLastError();
}

cudaError_t launch_group_advantage(int32_t B, int32_t G, const float* rewards, float* A_out,
                                   cudaStream_t s) {
  const int64_t groups = B / G;
  k_group_advantage<<<(unsigned)ceil_div(groups, 128), 128, 0, s>>>(B, G, rewards, A_out);
  return cudaGetLastError();
}

}  // namespace bgpo

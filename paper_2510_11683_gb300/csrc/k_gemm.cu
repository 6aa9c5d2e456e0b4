// The four LM-head contractions of the BGPO ELBO path on sm_103a tensor cores.
//
// Each is a persistent, warp-specialised kernel computing 128 x 256 fp32 tiles:
//   warp 0      TMA producer: 128-byte-swizzled bf16 tiles into a 4-stage ring
//   warp 1      TMEM owner + MMA issuer: tcgen05.mma kind::f16 (M=128, N=256,
//               K=16) into one of two TMEM accumulators (2 x 256 columns)
//   warps 2-5   epilogue: tcgen05.ld of the accumulator (thread = tile row),
//               fused per-kind epilogue, accumulator handed back to the MMA warp
// so the epilogue of tile n overlaps the main loop of tile n+1.
//
// Kinds (Xm = gathered masked hidden states [M, H], W = LM head [V, H]):
//   GEMM_FWD  z = Xm W^T; epilogue: online max / sum-exp per (row, vocab tile)
//             and the target logit (Eq. 4: log softmax gathered at y^i); full
//             logits are never written.
//   GEMM_DZ   z = Xm W^T recomputed; epilogue: dz = w_r (onehot - e^{z - lse})
//             stored as bf16 (gradient of Eq. 4 weighted by Eq. 13's dL/dl).
//   GEMM_DX   dXm = dZ W (K = vocabulary, split-K partials in fp32).
//   GEMM_DW   dW += dZ^T Xm (K = masked rows), fp32 read-modify-write.
//
// Every wait is bounded (time and polls); a wait that runs out sets the
// workspace error word to BGPO_ERR_TIMEOUT and the CTA drains and exits.
#include <math.h>

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

struct GemmParams {
  Geometry g;
  int num_sms;
  int32_t j;
  WsPtrs w;
  const float* coef;
  float* dW;
};

struct Work {
  int64_t units, tiles_m, tiles_n, kb_total;
  int splits;
};

struct Unit {
  int32_t m_blk, n_blk, split, kb0, kb_n;
};

template <int KIND>
__device__ __forceinline__ Work make_work(const GemmParams& p, int32_t M) {
  Work w;
  w.splits = 1;
  if (KIND == GEMM_FWD || KIND == GEMM_DZ) {
    w.tiles_m = ceil_div(M, kBM);
    w.tiles_n = p.g.n_vt;
    w.kb_total = p.g.H / kBK;
    w.units = w.tiles_m * w.tiles_n;
  } else if (KIND == GEMM_DX) {
    w.tiles_m = ceil_div(M, kBM);
    w.tiles_n = p.g.tiles_h;
    w.kb_total = p.g.kb_v;
    w.splits = w.tiles_m > 0 ? dx_splits(w.tiles_m, w.tiles_n, p.num_sms, w.kb_total,
                                         dxp_row_block_cap(p.g))
                             : 1;
    w.units = w.tiles_m * w.tiles_n * w.splits;
  } else {  // GEMM_DW
    w.tiles_m = ceil_div(p.g.V, kBM);
    w.tiles_n = p.g.tiles_h;
    w.kb_total = ceil_div(M, kBK);
    w.units = M > 0 ? w.tiles_m * w.tiles_n : 0;
  }
  return w;
}

template <int KIND>
__device__ __forceinline__ Unit unit_of(const Work& w, int64_t u) {
  Unit t;
  t.split = 0;
  if (KIND == GEMM_FWD || KIND == GEMM_DZ) {
    // consecutive units share a vocabulary tile of W: it is read from HBM once
    t.n_blk = (int32_t)(u / w.tiles_m);
    t.m_blk = (int32_t)(u % w.tiles_m);
    t.kb0 = 0;
    t.kb_n = (int32_t)w.kb_total;
  } else if (KIND == GEMM_DX) {
    const int64_t per_split = w.tiles_m * w.tiles_n;
    t.split = (int32_t)(u / per_split);
    const int64_t rem = u % per_split;
    t.n_blk = (int32_t)(rem / w.tiles_m);
    t.m_blk = (int32_t)(rem % w.tiles_m);
    const int64_t k0 = (int64_t)t.split * w.kb_total / w.splits;
    const int64_t k1 = (int64_t)(t.split + 1) * w.kb_total / w.splits;
    t.kb0 = (int32_t)k0;
    t.kb_n = (int32_t)(k1 - k0);
  } else {
    // consecutive units share a vocabulary block of dZ^T
    t.m_blk = (int32_t)(u / w.tiles_n);
    t.n_blk = (int32_t)(u % w.tiles_n);
    t.kb0 = 0;
    t.kb_n = (int32_t)w.kb_total;
  }
  return t;
}

template <int KIND>
struct Majors {
  static constexpr bool a_mn = (KIND == GEMM_DW);
  static constexpr bool b_mn = (KIND == GEMM_DX || KIND == GEMM_DW);
};

// Issues the TMA loads of one pipeline stage; returns the bytes they deliver.
template <int KIND>
__device__ __forceinline__ uint32_t load_stage(const GemmParams& p, const CUtensorMap* ma,
                                               const CUtensorMap* mb, uint32_t sa, uint32_t sb,
                                               uint32_t bar, const Unit& t, int32_t kb) {
  uint32_t bytes = 0;
  if (!Majors<KIND>::a_mn) {
    tma_load_2d(sa, ma, bar, kb * kBK, t.m_blk * kBM);
    bytes += kTileABytes;
  } else {
    // dZ^T tile: 2 boxes of 64 vocabulary columns x 64 masked rows
#pragma unroll
    for (int c = 0; c < kBM / 64; ++c) {
      const int32_t v = t.m_blk * kBM + c * 64;
      if (v < p.g.v_pad) {
        tma_load_2d(sa + c * kMnChunkBytes, ma, bar, v, kb * kBK);
        bytes += kMnChunkBytes;
      }
    }
  }
  if (!Majors<KIND>::b_mn) {
    tma_load_2d(sb, mb, bar, kb * kBK, t.n_blk * kBN);
    bytes += kTileBBytes;
  } else {
    // W (GEMM_DX) or Xm (GEMM_DW) tile: 4 boxes of 64 hidden columns x 64 K rows
#pragma unroll
    for (int c = 0; c < kBN / 64; ++c) {
      const int32_t h = t.n_blk * kBN + c * 64;
      if (h < p.g.H) {
        tma_load_2d(sb + c * kMnChunkBytes, mb, bar, h, kb * kBK);
        bytes += kMnChunkBytes;
      }
    }
  }
  return bytes;
}

__device__ __forceinline__ float bits_f(uint32_t v) { return __uint_as_float(v); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// ---- epilogues: one thread per accumulator row ----------------------------------

// GEMM_FWD: per (row, vocab tile) the pair (max z, sum e^{z - max}) and, in the
// tile holding y_r, the target logit z_{r, y_r}.
__device__ __forceinline__ void epi_fwd(const GemmParams& p, int32_t M, const Unit& t, int row,
                                        uint32_t tb) {
  const int64_t r = (int64_t)t.m_blk * kBM + row;
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
    float cm = -INFINITY;
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      const float z = bits_f(raw[k]);
      if (k < nvalid) cm = fmaxf(cm, z);
      if (col0 + k == y) { tl = z; hit = true; }
    }
    const float mn = fmaxf(m, cm);
    const float mnl = mn * kLog2e;
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < 32; ++k)
      if (k < nvalid) acc += exp2f(fmaf(bits_f(raw[k]), kLog2e, -mnl));
    s = s * exp2f((m - mn) * kLog2e) + acc;
    m = mn;
  }
  if (valid) {
    p.w.part[r * p.g.n_vt + t.n_blk] = make_float2(m, s);
    if (hit) p.w.tgt_logit[r] = tl;
  }
}

// GEMM_DZ: dz_{r,v} = w_r (1[v = y_r] - e^{z_{r,v} - lse_r}) as bf16, zero for
// rows >= M and vocabulary columns >= V (the dZ row pitch is v_pad).
__device__ __forceinline__ void epi_dz(const GemmParams& p, int32_t M, const Unit& t, int row,
                                       uint32_t tb) {
  const int64_t r = (int64_t)t.m_blk * kBM + row;
  const bool valid = r < M;
  float w = 0.f, lse_l2 = 0.f;
  int32_t y = -1;
  if (valid) {
    const int32_t b = p.w.rows[r] / (int32_t)p.g.R;
    w = p.coef[b] / p.w.t[b];
    lse_l2 = p.w.lse[r] * kLog2e;
    y = p.w.tgt[r];
  }
  const int32_t v0 = t.n_blk * kBN;
  const int32_t V = (int32_t)p.g.V;
  __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(p.w.dz) + r * p.g.v_pad + v0;
#pragma unroll 1
  for (int c = 0; c < kBN / 32; ++c) {
    const int32_t col0 = v0 + c * 32;
    if (col0 >= p.g.v_pad) break;  // warp-uniform
    uint32_t raw[32];
    tmem_ld_32x32b_x32(tb + c * 32, raw);
    tmem_ld_wait();
    uint32_t packed[16];
#pragma unroll
    for (int k = 0; k < 32; k += 2) {
      float d[2];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int32_t col = col0 + k + e;
        const float pr = exp2f(fmaf(bits_f(raw[k + e]), kLog2e, -lse_l2));
        const float v = w * ((col == y ? 1.f : 0.f) - pr);
        d[e] = (valid && col < V) ? v : 0.f;
      }
      packed[k / 2] = pack_bf16x2(d[0], d[1]);
    }
    uint4* o = reinterpret_cast<uint4*>(dst + c * 32);
#pragma unroll
    for (int q = 0; q < 4; ++q)
      o[q] = make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2], packed[4 * q + 3]);
  }
}

// GEMM_DX: fp32 partial of split s for masked row r.
__device__ __forceinline__ void epi_dx(const GemmParams& p, int32_t M, const Work& wk, const Unit& t,
                                       int row, uint32_t tb) {
  const int64_t r = (int64_t)t.m_blk * kBM + row;
  const int32_t h0 = t.n_blk * kBN;
  const int64_t split_stride = wk.tiles_m * kBM * p.g.H;
  float* dst = p.w.dxp + t.split * split_stride + r * p.g.H + h0;
#pragma unroll 1
  for (int c = 0; c < kBN / 32; ++c) {
    if (h0 + c * 32 >= p.g.H) break;  // warp-uniform
    uint32_t raw[32];
    tmem_ld_32x32b_x32(tb + c * 32, raw);
    tmem_ld_wait();
    if (r < M) {
      float4* o = reinterpret_cast<float4*>(dst + c * 32);
#pragma unroll
      for (int q = 0; q < 8; ++q)
        o[q] = make_float4(bits_f(raw[4 * q]), bits_f(raw[4 * q + 1]), bits_f(raw[4 * q + 2]),
                           bits_f(raw[4 * q + 3]));
    }
  }
}

// GEMM_DW: dW[v, h] += acc for vocabulary row v < V.
__device__ __forceinline__ void epi_dw(const GemmParams& p, const Unit& t, int row, uint32_t tb) {
  const int64_t v = (int64_t)t.m_blk * kBM + row;
  const int32_t h0 = t.n_blk * kBN;
  float* dst = p.dW + v * p.g.H + h0;
#pragma unroll 1
  for (int c = 0; c < kBN / 32; ++c) {
    if (h0 + c * 32 >= p.g.H) break;  // warp-uniform
    uint32_t raw[32];
    tmem_ld_32x32b_x32(tb + c * 32, raw);
    tmem_ld_wait();
    if (v < p.g.V) {
      float4* o = reinterpret_cast<float4*>(dst + c * 32);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        float4 a = o[q];
        a.x += bits_f(raw[4 * q]);
        a.y += bits_f(raw[4 * q + 1]);
        a.z += bits_f(raw[4 * q + 2]);
        a.w += bits_f(raw[4 * q + 3]);
        o[q] = a;
      }
    }
  }
}

template <int KIND>
__device__ __forceinline__ int32_t kernel_id() {
  return KIND == GEMM_FWD ? KID_LMHEAD_FWD
       : KIND == GEMM_DZ  ? KID_LMHEAD_DZ
       : KIND == GEMM_DX  ? KID_DX_GEMM
                          : KID_DW_GEMM;
}

template <int KIND>
__global__ void __launch_bounds__(kThreads, 1)
    k_gemm(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
           const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* s_a = smem;
  uint8_t* s_b = smem + kStages * kTileABytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_b + kStages * kTileBBytes);
  uint64_t* full = bars;                      // [kStages] TMA -> MMA
  uint64_t* empty = bars + kStages;           // [kStages] MMA -> TMA
  uint64_t* tfull = bars + 2 * kStages;       // [2] MMA -> epilogue
  uint64_t* tempty = bars + 2 * kStages + 2;  // [2] epilogue -> MMA
  uint64_t* done = bars + 2 * kStages + 4;    // MMA drain on abort
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kStages + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* never = reinterpret_cast<volatile int*>(tmem_slot + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  int32_t* err = p.w.err;

  int32_t M = 0;
  if (err[ERR_SAMPLE] == p.j) {
    M = err[ERR_M];
  } else if (blockIdx.x == 0 && threadIdx.x == 0) {
    set_device_error(err, kStatusInvalidArg, kernel_id<KIND>() * 16 + 1);
  }
  const Work wk = make_work<KIND>(p, M);
  if ((int64_t)blockIdx.x >= wk.units) return;  // whole CTA, before any allocation

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_addr(&full[s]), 1);
      mbar_init(smem_addr(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_addr(&tfull[a]), 1);
      mbar_init(smem_addr(&tempty[a]), 4 * 32);
    }
    mbar_init(smem_addr(done), 1);
    *abort_flag = 0;
    *never = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&map_a);
    tma_prefetch_map(&map_b);
  }
  if (warp == 1) {
    tmem_alloc(smem_addr(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      uint32_t armed = 0;  // bit s: stage s has copies that may still be in flight
      for (int64_t u = blockIdx.x; u < wk.units && ok; u += gridDim.x) {
        const Unit t = unit_of<KIND>(wk, u);
        for (int32_t kb = t.kb0; kb < t.kb0 + t.kb_n; ++kb) {
          if (!mbar_wait(smem_addr(&empty[stage]), phase ^ 1u, abort_flag)) { ok = false; break; }
          const uint32_t bar = smem_addr(&full[stage]);
          const uint32_t sa = smem_addr(s_a + stage * kTileABytes);
          const uint32_t sb = smem_addr(s_b + stage * kTileBBytes);
          // the expected byte count is armed before the copies that complete it
          uint32_t bytes = 0;
          if (!Majors<KIND>::a_mn) bytes += kTileABytes;
          else
            for (int c = 0; c < kBM / 64; ++c)
              if (t.m_blk * kBM + c * 64 < p.g.v_pad) bytes += kMnChunkBytes;
          if (!Majors<KIND>::b_mn) bytes += kTileBBytes;
          else
            for (int c = 0; c < kBN / 64; ++c)
              if (t.n_blk * kBN + c * 64 < p.g.H) bytes += kMnChunkBytes;
          mbar_arrive_expect_tx(bar, bytes);
          load_stage<KIND>(p, &map_a, &map_b, sa, sb, bar, t, kb);
          armed |= 1u << stage;
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
      }
      if (!ok) {
        *abort_flag = 1;
        set_device_error(err, kStatusTimeout, kernel_id<KIND>() * 16 + 2);
        // Let copies already issued land before the CTA exits: stage s was last
        // armed in phase `phase` if s < stage, else in phase `phase ^ 1`.
        for (int s = 0; s < kStages; ++s) {
          if (!((armed >> s) & 1u)) continue;
          const uint32_t ph = (s < stage) ? phase : (phase ^ 1u);
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(smem_addr(&full[s]), ph) && globaltimer_ns() - t0 < 10000000ull) {
          }
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, kBN, Majors<KIND>::a_mn, Majors<KIND>::b_mn);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true, issued = false;
      int it = 0;
      for (int64_t u = blockIdx.x; u < wk.units && ok; u += gridDim.x, ++it) {
        const Unit t = unit_of<KIND>(wk, u);
        const int acc = it & 1;
        const uint32_t acc_phase = (uint32_t)(it >> 1) & 1u;
        if (!mbar_wait(smem_addr(&tempty[acc]), acc_phase ^ 1u, abort_flag)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * kBN);
        for (int32_t kb = 0; kb < t.kb_n; ++kb) {
          if (!mbar_wait(smem_addr(&full[stage]), phase, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sa = smem_addr(s_a + stage * kTileABytes);
          const uint32_t sb = smem_addr(s_b + stage * kTileBBytes);
#pragma unroll
          for (int k = 0; k < kBK / kUmmaK; ++k) {
            const uint64_t ad = Majors<KIND>::a_mn ? smem_desc_sw128(sa + k * 2048, kMnChunkBytes, 1024)
                                                   : smem_desc_sw128(sa + k * 32, 16, 1024);
            const uint64_t bd = Majors<KIND>::b_mn ? smem_desc_sw128(sb + k * 2048, kMnChunkBytes, 1024)
                                                   : smem_desc_sw128(sb + k * 32, 16, 1024);
            umma_bf16(d_tmem, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          }
          issued = true;
          umma_commit(smem_addr(&empty[stage]));  // frees the stage once these MMAs finish
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        umma_commit(smem_addr(&tfull[acc]));  // accumulator ready for the epilogue
      }
      if (!ok) {
        *abort_flag = 1;
        set_device_error(err, kStatusTimeout, kernel_id<KIND>() * 16 + 3);
        if (issued) {
          umma_commit(smem_addr(done));
          mbar_wait(smem_addr(done), 0, never);
        }
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue (warps 2..5) ----------------
    const int quarter = warp & 3;  // TMEM lanes this warp may access: 32*quarter ..
    const int row = quarter * 32 + lane;
    int it = 0;
    bool ok = true;
    for (int64_t u = blockIdx.x; u < wk.units; u += gridDim.x, ++it) {
      const Unit t = unit_of<KIND>(wk, u);
      const int acc = it & 1;
      const uint32_t acc_phase = (uint32_t)(it >> 1) & 1u;
      const bool got = mbar_wait(smem_addr(&tfull[acc]), acc_phase, abort_flag);
      if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
      tc_fence_after();
      const uint32_t tb = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * kBN);
      if (KIND == GEMM_FWD) epi_fwd(p, M, t, row, tb);
      else if (KIND == GEMM_DZ) epi_dz(p, M, t, row, tb);
      else if (KIND == GEMM_DX) epi_dx(p, M, wk, t, row, tb);
      else epi_dw(p, t, row, tb);
      tc_fence_before();
      mbar_arrive(smem_addr(&tempty[acc]));
    }
    if (!ok) {
      *abort_flag = 1;
      if (lane == 0) set_device_error(err, kStatusTimeout, kernel_id<KIND>() * 16 + 4);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

template <int KIND>
cudaError_t launch_kind(const CUtensorMap& ma, const CUtensorMap& mb, const GemmParams& p,
                        cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(k_gemm<KIND>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kGemmSmemBytes);
  if (e != cudaSuccess) return e;
  k_gemm<KIND><<<p.num_sms, kThreads, kGemmSmemBytes, s>>>(ma, mb, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm(GemmKind kind, const CUtensorMap& map_a, const CUtensorMap& map_b,
                        const GemmArgs& a, const WsPtrs& w, cudaStream_t s) {
  GemmParams p;
  p.g = a.g;
  p.num_sms = a.num_sms;
  p.j = a.j;
  p.w = w;
  p.coef = a.coef;
  p.dW = a.dW;
  switch (kind) {
    case GEMM_FWD: return launch_kind<GEMM_FWD>(map_a, map_b, p, s);
    case GEMM_DZ: return launch_kind<GEMM_DZ>(map_a, map_b, p, s);
    case GEMM_DX: return launch_kind<GEMM_DX>(map_a, map_b, p, s);
    case GEMM_DW: return launch_kind<GEMM_DW>(map_a, map_b, p, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace bgpo

// Host side of the C ABI declared in include/bgpo.h: argument validation,
// workspace layout, TMA tensor-map encoding, kernel launches, per-kernel
// event tracing and an NVTX range named after each launching call. Keeps no state between calls except the cached driver entry
// point of cuTensorMapEncodeTiled.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <nvtx3/nvToolsExt.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include <mutex>

#include "bgpo.h"
#include "bgpo_internal.h"
#include "bgpo_plan.h"

using namespace bgpo;

struct bgpo_trace {
  int32_t capacity;
  int32_t count;
  int32_t* ids;
  cudaEvent_t* start;
  cudaEvent_t* stop;
};

namespace {

constexpr int64_t kMaxRows = int64_t(1) << 22;  // B * R
constexpr int64_t kMaxV = int64_t(1) << 24;
constexpr int64_t kMaxH = 16384;

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Records CUDA events around one kernel launch when a trace is attached.
struct TraceScope {
  bgpo_trace* tr;
  cudaStream_t s;
  int32_t idx;
  TraceScope(bgpo_trace* t, int32_t kid, cudaStream_t st) : tr(t), s(st), idx(-1) {
    if (tr && tr->count < tr->capacity) {
      idx = tr->count++;
      tr->ids[idx] = kid;
      cudaEventRecord(tr->start[idx], s);
    }
  }
  ~TraceScope() {
    if (idx >= 0) cudaEventRecord(tr->stop[idx], s);
  }
};

// NVTX range around one launching C-ABI call, named after it (shows in Nsight
// timelines; a no-op when no tool is attached).
struct CallRange {
  explicit CallRange(const char* name) { nvtxRangePushA(name); }
  ~CallRange() { nvtxRangePop(); }
  CallRange(const CallRange&) = delete;
  CallRange& operator=(const CallRange&) = delete;
};

bgpo_status check_problem(const bgpo_problem* p) {
  if (!p) return BGPO_ERR_INVALID_ARG;
  if (p->t_mode != BGPO_T_IID && p->t_mode != BGPO_T_STRATIFIED) return BGPO_ERR_INVALID_ARG;
  if (p->b_offset < 0) return BGPO_ERR_INVALID_ARG;
  if (!isfinite(p->loss_scale)) return BGPO_ERR_INVALID_ARG;
  if ((p->flags & ~(BGPO_FLAG_KEEP_LOGITS | BGPO_FLAG_PAIR_DW)) != 0u) return BGPO_ERR_INVALID_ARG;
  if (p->vocab_chunk < 0 || p->vocab_chunk % kBN != 0) return BGPO_ERR_INVALID_ARG;
  if (p->B < 1 || p->P < 0 || p->R < 1 || p->V < 1 || p->n_t < 1 || p->G < 1) return BGPO_ERR_SHAPE;
  if (p->H < 64 || p->H % 8 != 0 || p->H > kMaxH) return BGPO_ERR_SHAPE;
  if (p->V > kMaxV || p->n_t >= 65536) return BGPO_ERR_SHAPE;
  if ((int64_t)p->B * p->R > kMaxRows) return BGPO_ERR_SHAPE;
  if ((int64_t)p->b_offset + p->B > (int64_t(1) << 31)) return BGPO_ERR_SHAPE;
  if ((int64_t)p->B * ((int64_t)p->P + p->R) * p->H > (int64_t(1) << 40)) return BGPO_ERR_SHAPE;
  return BGPO_OK;
}

bool keeps_logits(const bgpo_problem* p) { return (p->flags & BGPO_FLAG_KEEP_LOGITS) != 0u; }

bool pairs_dw(const bgpo_problem* p) { return (p->flags & BGPO_FLAG_PAIR_DW) != 0u; }

Geometry geometry_of(const bgpo_problem* p) {
  return make_geometry(p->B, p->P, p->R, p->H, p->V, p->vocab_chunk, pairs_dw(p));
}

bgpo_status check_sample(const bgpo_problem* p, int32_t j) {
  return (j >= 0 && j < p->n_t) ? BGPO_OK : BGPO_ERR_INVALID_ARG;
}

bgpo_status check_ws(const bgpo_problem* p, const void* ws, size_t ws_bytes, WsLayout* L) {
  if (!ws) return BGPO_ERR_INVALID_ARG;
  if (!aligned(ws, 256)) return BGPO_ERR_ALIGNMENT;
  *L = make_ws_layout(geometry_of(p), keeps_logits(p), pairs_dw(p));
  if (ws_bytes < L->total) return BGPO_ERR_WORKSPACE_TOO_SMALL;
  return BGPO_OK;
}

bgpo_status device_sms(int* num_sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return BGPO_ERR_UNSUPPORTED_DEVICE;
  }
  int major = 0, minor = 0, sms = 0;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return BGPO_ERR_CUDA;
  }
  if (major != 10 || minor != 3) return BGPO_ERR_UNSUPPORTED_DEVICE;
  *num_sms = sms;
  return BGPO_OK;
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(f);
    else
      cudaGetLastError();
  });
  return fn;
}

// 2-D tensor map over a row-major [outer, inner] matrix with row pitch
// `pitch_bytes`, 128-byte swizzle, zero fill outside the matrix (bf16 by
// default, fp32 for the fp32 epilogue destinations).
bool map_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t pitch_bytes,
            uint32_t box_inner, uint32_t box_outer,
            CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16) {
  EncodeTiledFn enc = encode_tiled();
  if (!enc) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {pitch_bytes};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, dtype, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bgpo_status from_cuda(cudaError_t e) { return e == cudaSuccess ? BGPO_OK : BGPO_ERR_CUDA; }

}  // namespace

extern "C" {

int32_t bgpo_abi_version(void) { return BGPO_ABI_VERSION; }

const char* bgpo_status_string(bgpo_status s) {
  switch (s) {
    case BGPO_OK: return "BGPO_OK";
    case BGPO_ERR_INVALID_ARG: return "BGPO_ERR_INVALID_ARG";
    case BGPO_ERR_SHAPE: return "BGPO_ERR_SHAPE";
    case BGPO_ERR_ALIGNMENT: return "BGPO_ERR_ALIGNMENT";
    case BGPO_ERR_WORKSPACE_TOO_SMALL: return "BGPO_ERR_WORKSPACE_TOO_SMALL";
    case BGPO_ERR_NONFINITE: return "BGPO_ERR_NONFINITE";
    case BGPO_ERR_UNSUPPORTED_DEVICE: return "BGPO_ERR_UNSUPPORTED_DEVICE";
    case BGPO_ERR_CUDA: return "BGPO_ERR_CUDA";
    case BGPO_ERR_TIMEOUT: return "BGPO_ERR_TIMEOUT";
    case BGPO_ERR_BOUNDS: return "BGPO_ERR_BOUNDS";
  }
  return "BGPO_ERR_UNKNOWN";
}

bgpo_status bgpo_validate_problem(const bgpo_problem* prob) { return check_problem(prob); }

size_t bgpo_workspace_bytes(const bgpo_problem* prob) {
  if (check_problem(prob) != BGPO_OK) return 0;
  return make_ws_layout(geometry_of(prob), keeps_logits(prob), pairs_dw(prob)).total;
}

bgpo_status bgpo_sample_mask(const bgpo_problem* prob, int32_t j, void* ws, size_t ws_bytes,
                             float* t_out, uint8_t* mask_out, void* stream) {
  CallRange range("bgpo_sample_mask");
  bgpo_status st = check_problem(prob);
  if (st != BGPO_OK) return st;
  if ((st = check_sample(prob, j)) != BGPO_OK) return st;
  WsLayout L;
  if ((st = check_ws(prob, ws, ws_bytes, &L)) != BGPO_OK) return st;
  if ((t_out && !aligned(t_out, 4)) || (prob->resp_len && !aligned(prob->resp_len, 4)))
    return BGPO_ERR_ALIGNMENT;
  int sms = 0;
  if ((st = device_sms(&sms)) != BGPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const WsPtrs w = ws_pointers(ws, L);
  MaskArgs a;
  a.seed = prob->seed;
  a.b_offset = prob->b_offset;
  a.B = prob->B;
  a.R = prob->R;
  a.j = j;
  a.n_t = prob->n_t;
  a.t_mode = prob->t_mode;
  a.t_out = t_out;
  a.mask_out = mask_out;
  a.resp_len = prob->resp_len;
  a.pair_dw = pairs_dw(prob);
  TraceScope ts(prob->trace, KID_MASK_COMPACT, s);
  return from_cuda(launch_mask_compact(a, w, s));
}

bgpo_status bgpo_elbo_fwd(const bgpo_problem* prob, int32_t j, const void* X, const void* W,
                          const int32_t* Y, void* ws, size_t ws_bytes, float* ell_out,
                          void* stream) {
  CallRange range("bgpo_elbo_fwd");
  bgpo_status st = check_problem(prob);
  if (st != BGPO_OK) return st;
  if ((st = check_sample(prob, j)) != BGPO_OK) return st;
  if (!X || !W || !Y || !ell_out) return BGPO_ERR_INVALID_ARG;
  if (!aligned(X, 16) || !aligned(W, 16) || !aligned(Y, 4) || !aligned(ell_out, 4))
    return BGPO_ERR_ALIGNMENT;
  WsLayout L;
  if ((st = check_ws(prob, ws, ws_bytes, &L)) != BGPO_OK) return st;
  int sms = 0;
  if ((st = device_sms(&sms)) != BGPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const Geometry g = geometry_of(prob);
  const WsPtrs w = ws_pointers(ws, L);

  const bool keep = w.zc != nullptr;
  CUtensorMap map_xm, map_w, map_zc;
  if (!map_2d(&map_xm, w.xm, g.H, g.m_pad, g.H * 2, kBK, kBM) ||
      !map_2d(&map_w, W, g.H, g.V, g.H * 2, kBK, kBNHalf) ||
      // logits leave the epilogue as 32-row x 32-column fp32 sub-tiles
      (keep && !map_2d(&map_zc, w.zc, g.v_pad, g.m_pad, g.v_pad * 4, 32, 32,
                       CU_TENSOR_MAP_DATA_TYPE_FLOAT32)))
    return BGPO_ERR_CUDA;
  GemmArgs ga;
  ga.g = g;
  ga.num_pairs = gemm_num_pairs(sms);
  ga.j = j;
  ga.coef = nullptr;
  ga.dW = nullptr;
  {
    TraceScope ts(prob->trace, KID_GATHER, s);
    if (launch_gather(g, j, X, Y, w, s) != cudaSuccess) return BGPO_ERR_CUDA;
  }
  {
    TraceScope ts(prob->trace, KID_LMHEAD_FWD, s);
    if (launch_gemm(GEMM_FWD, map_xm, map_w, keep ? map_zc : map_xm, ga, w, s) != cudaSuccess)
      return BGPO_ERR_CUDA;
  }
  {
    TraceScope ts(prob->trace, KID_LSE_COMBINE, s);
    if (launch_lse_combine(g, j, keep, w, s) != cudaSuccess) return BGPO_ERR_CUDA;
  }
  {
    TraceScope ts(prob->trace, KID_SEQ_REDUCE, s);
    if (launch_seq_reduce(g, j, w, ell_out, s) != cudaSuccess) return BGPO_ERR_CUDA;
  }
  return BGPO_OK;
}

bgpo_status bgpo_bound_coeffs(const bgpo_problem* prob, int32_t j, const float* ell,
                              const float* ell_old, const float* A, float* coef_out, float* g_out,
                              void* ws, size_t ws_bytes, void* stream) {
  CallRange range("bgpo_bound_coeffs");
  bgpo_status st = check_problem(prob);
  if (st != BGPO_OK) return st;
  if ((st = check_sample(prob, j)) != BGPO_OK) return st;
  if (!ell || !ell_old || !A || !coef_out) return BGPO_ERR_INVALID_ARG;
  if (!aligned(ell, 4) || !aligned(ell_old, 4) || !aligned(A, 4) || !aligned(coef_out, 4) ||
      (g_out && !aligned(g_out, 4)))
    return BGPO_ERR_ALIGNMENT;
  WsLayout L;
  if ((st = check_ws(prob, ws, ws_bytes, &L)) != BGPO_OK) return st;
  int sms = 0;
  if ((st = device_sms(&sms)) != BGPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const WsPtrs w = ws_pointers(ws, L);
  TraceScope ts(prob->trace, KID_BOUND_COEFFS, s);
  return from_cuda(launch_bound_coeffs(prob->B, prob->n_t, prob->loss_scale, ell, ell_old, A,
                                       coef_out, g_out, w, s));
}

bgpo_status bgpo_vrpo_coeffs(const bgpo_problem* prob, const float* ell, const float* ell_old,
                             const float* A, float* coef_out, float* R_out, void* ws,
                             size_t ws_bytes, void* stream) {
  CallRange range("bgpo_vrpo_coeffs");
  bgpo_status st = check_problem(prob);
  if (st != BGPO_OK) return st;
  if (!ell || !ell_old || !A || !coef_out) return BGPO_ERR_INVALID_ARG;
  if (!aligned(ell, 4) || !aligned(ell_old, 4) || !aligned(A, 4) || !aligned(coef_out, 4) ||
      (R_out && !aligned(R_out, 4)))
    return BGPO_ERR_ALIGNMENT;
  WsLayout L;
  if ((st = check_ws(prob, ws, ws_bytes, &L)) != BGPO_OK) return st;
  int sms = 0;
  if ((st = device_sms(&sms)) != BGPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const WsPtrs w = ws_pointers(ws, L);
  TraceScope ts(prob->trace, KID_VRPO_COEFFS, s);
  return from_cuda(launch_vrpo_coeffs(prob->B, prob->n_t, prob->loss_scale, ell, ell_old, A,
                                      coef_out, R_out, w, s));
}

bgpo_status bgpo_elbo_bwd_accumulate(const bgpo_problem* prob, int32_t j, const void* X,
                                     const void* W, const int32_t* Y, const float* coef, void* ws,
                                     size_t ws_bytes, float* dX, float* dW, void* stream) {
  CallRange range("bgpo_elbo_bwd_accumulate");
  bgpo_status st = check_problem(prob);
  if (st != BGPO_OK) return st;
  if ((st = check_sample(prob, j)) != BGPO_OK) return st;
  if (!X || !W || !Y || !coef || !dX || !dW) return BGPO_ERR_INVALID_ARG;
  if (!aligned(X, 16) || !aligned(W, 16) || !aligned(Y, 4) || !aligned(coef, 4) ||
      !aligned(dX, 16) || !aligned(dW, 16))
    return BGPO_ERR_ALIGNMENT;
  WsLayout L;
  if ((st = check_ws(prob, ws, ws_bytes, &L)) != BGPO_OK) return st;
  int sms = 0;
  if ((st = device_sms(&sms)) != BGPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const Geometry g = geometry_of(prob);
  const WsPtrs w = ws_pointers(ws, L);

  const bool keep = w.zc != nullptr;
  // dW pairing: an even sample's dW GEMM waits for the next sample's (unless it
  // is the last sample); an odd sample's dW GEMM covers both samples' rows
  const bool pair = pairs_dw(prob);
  const bool defer = pair && j % 2 == 0 && j + 1 < prob->n_t;
  const uint64_t zr = (uint64_t)w.dz_rows;
  const uint64_t zc = (uint64_t)w.dz_cols;
  CUtensorMap map_xm_k, map_w_k, map_dz_k, map_w_mn, map_dz_mn, map_xmT_k;
  CUtensorMap map_dz_st, map_dxp_st, map_dw_red;
  const uint64_t dxp_rows = (uint64_t)dxp_row_block_cap(g) * kPairM;
  if (!map_2d(&map_xm_k, w.xm, g.H, g.m_pad, g.H * 2, kBK, kBM) ||
      !map_2d(&map_w_k, W, g.H, g.V, g.H * 2, kBK, kBNHalf) ||
      !map_2d(&map_dz_k, w.dz, zc, zr, zc * 2, kBK, kBM) ||
      !map_2d(&map_w_mn, W, g.H, g.V, g.H * 2, 64, kBK) ||
      !map_2d(&map_dz_mn, w.dz, zc, zr, zc * 2, 64, kBK) ||
      !map_2d(&map_xmT_k, w.xmT, zr, g.H, zr * 2, kBK, kBNHalf) ||
      // epilogue destinations: 32-row sub-tiles of 128 bytes
      !map_2d(&map_dz_st, w.dz, zc, zr, zc * 2, 64, 32) ||
      !map_2d(&map_dxp_st, w.dxp, g.H, dxp_rows, g.H * 4, 32, 32, CU_TENSOR_MAP_DATA_TYPE_FLOAT32) ||
      !map_2d(&map_dw_red, dW, g.H, g.V, g.H * 4, 32, 32, CU_TENSOR_MAP_DATA_TYPE_FLOAT32))
    return BGPO_ERR_CUDA;
  GemmArgs ga;
  ga.g = g;
  ga.num_pairs = gemm_num_pairs(sms);
  ga.j = j;
  ga.coef = coef;
  ga.dW = dW;
  ga.dX = dX;
  ga.pair_consume = pair && (j & 1);
  {
    // Xm^T for the dW GEMMs; also records the dW pairing state of this sample
    TraceScope ts(prob->trace, KID_XM_TRANSPOSE, s);
    if (launch_xm_transpose(g, j, defer, w, s) != cudaSuccess) return BGPO_ERR_CUDA;
  }
  // One vocabulary chunk at a time (Linearity, Sec. 3, within a sample: the
  // gradient is a sum over vocabulary entries too): dZ of the chunk, its dX
  // contribution, and, when dZ holds one chunk, the chunk's rows of dW.
  for (int64_t c = 0; c < g.n_vc; ++c) {
    ga.v_begin = chunk_begin(g, c);
    ga.v_end = chunk_end(g, c);
    ga.dz_col0 = w.dz_chunk_local ? 0 : ga.v_begin;
    ga.chunk = c;
    if (keep) {
      TraceScope ts(prob->trace, KID_DZ_FROM_LOGITS, s);
      if (launch_dz_from_logits(g, j, c, coef, sms, w, s) != cudaSuccess) return BGPO_ERR_CUDA;
    } else {
      TraceScope ts(prob->trace, KID_LMHEAD_DZ, s);
      if (launch_gemm(GEMM_DZ, map_xm_k, map_w_k, map_dz_st, ga, w, s) != cudaSuccess)
        return BGPO_ERR_CUDA;
    }
    {
      TraceScope ts(prob->trace, KID_DX_GEMM, s);
      if (launch_gemm(GEMM_DX, map_dz_k, map_w_mn, map_dxp_st, ga, w, s) != cudaSuccess)
        return BGPO_ERR_CUDA;
    }
    if (w.dz_chunk_local) {
      TraceScope ts(prob->trace, KID_DW_GEMM, s);
      if (launch_gemm(GEMM_DW, map_dz_mn, map_xmT_k, map_dw_red, ga, w, s) != cudaSuccess)
        return BGPO_ERR_CUDA;
    }
  }
  {
    TraceScope ts(prob->trace, KID_DX_REDUCE, s);
    if (launch_dx_reduce(g, j, w, dX, s) != cudaSuccess) return BGPO_ERR_CUDA;
  }
  if (!w.dz_chunk_local && !defer) {
    // dZ spans the whole vocabulary (one chunk, or dW pairing): one dW GEMM
    ga.v_begin = 0;
    ga.v_end = g.V;
    ga.dz_col0 = 0;
    TraceScope ts(prob->trace, KID_DW_GEMM, s);
    if (launch_gemm(GEMM_DW, map_dz_mn, map_xmT_k, map_dw_red, ga, w, s) != cudaSuccess)
      return BGPO_ERR_CUDA;
  }
  return BGPO_OK;
}

bgpo_status bgpo_group_advantage(const bgpo_problem* prob, const float* rewards, float* A_out,
                                 void* stream) {
  CallRange range("bgpo_group_advantage");
  bgpo_status st = check_problem(prob);
  if (st != BGPO_OK) return st;
  if (!rewards || !A_out) return BGPO_ERR_INVALID_ARG;
  if (prob->B % prob->G != 0) return BGPO_ERR_SHAPE;
  if (!aligned(rewards, 4) || !aligned(A_out, 4)) return BGPO_ERR_ALIGNMENT;
  int sms = 0;
  if ((st = device_sms(&sms)) != BGPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  TraceScope ts(prob->trace, KID_GROUP_ADV, s);
  return from_cuda(launch_group_advantage(prob->B, prob->G, rewards, A_out, s));
}

bgpo_status bgpo_get_device_error(const void* ws, size_t ws_bytes, int32_t* code_out,
                                  int32_t* where_out, void* stream) {
  if (!ws || !code_out) return BGPO_ERR_INVALID_ARG;
  if (!aligned(ws, 256)) return BGPO_ERR_ALIGNMENT;
  if (ws_bytes < 64) return BGPO_ERR_WORKSPACE_TOO_SMALL;
  int32_t host[2] = {0, 0};
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(host, ws, sizeof(host), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return BGPO_ERR_CUDA;
  }
  *code_out = host[ERR_STATUS];
  if (where_out) *where_out = host[ERR_WHERE];
  return BGPO_OK;
}

bgpo_status bgpo_clear_device_error(void* ws, size_t ws_bytes, void* stream) {
  if (!ws) return BGPO_ERR_INVALID_ARG;
  if (!aligned(ws, 256)) return BGPO_ERR_ALIGNMENT;
  if (ws_bytes < 64) return BGPO_ERR_WORKSPACE_TOO_SMALL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // status and where to 0; the dW pairing state (ERR_PEND .. ERR_PAIRED) to -1:
  // nothing pending
  if (cudaMemsetAsync(ws, 0, 2 * sizeof(int32_t), s) != cudaSuccess ||
      cudaMemsetAsync(static_cast<int32_t*>(ws) + ERR_PEND, 0xff, 4 * sizeof(int32_t), s) !=
          cudaSuccess) {
    cudaGetLastError();
    return BGPO_ERR_CUDA;
  }
  return BGPO_OK;
}

bgpo_status bgpo_selftest_bounded_wait(void* ws, size_t ws_bytes, uint32_t timeout_us,
                                       void* stream) {
  if (!ws) return BGPO_ERR_INVALID_ARG;
  if (!aligned(ws, 256)) return BGPO_ERR_ALIGNMENT;
  if (ws_bytes < 64) return BGPO_ERR_WORKSPACE_TOO_SMALL;
  if (timeout_us == 0 || timeout_us > 1000000u) return BGPO_ERR_INVALID_ARG;
  int sms = 0;
  bgpo_status st = device_sms(&sms);
  if (st != BGPO_OK) return st;
  return from_cuda(launch_selftest_wait(static_cast<int32_t*>(ws), (uint64_t)timeout_us * 1000ull,
                                        static_cast<cudaStream_t>(stream)));
}

bgpo_trace* bgpo_trace_create(int32_t capacity) {
  if (capacity <= 0) return nullptr;
  bgpo_trace* t = static_cast<bgpo_trace*>(calloc(1, sizeof(bgpo_trace)));
  if (!t) return nullptr;
  t->capacity = capacity;
  t->ids = static_cast<int32_t*>(calloc((size_t)capacity, sizeof(int32_t)));
  t->start = static_cast<cudaEvent_t*>(calloc((size_t)capacity, sizeof(cudaEvent_t)));
  t->stop = static_cast<cudaEvent_t*>(calloc((size_t)capacity, sizeof(cudaEvent_t)));
  bool ok = t->ids && t->start && t->stop;
  for (int32_t i = 0; ok && i < capacity; ++i)
    ok = cudaEventCreate(&t->start[i]) == cudaSuccess && cudaEventCreate(&t->stop[i]) == cudaSuccess;
  if (!ok) {
    cudaGetLastError();
    bgpo_trace_destroy(t);
    return nullptr;
  }
  return t;
}

void bgpo_trace_destroy(bgpo_trace* t) {
  if (!t) return;
  for (int32_t i = 0; i < t->capacity; ++i) {
    if (t->start && t->start[i]) cudaEventDestroy(t->start[i]);
    if (t->stop && t->stop[i]) cudaEventDestroy(t->stop[i]);
  }
  free(t->ids);
  free(t->start);
  free(t->stop);
  free(t);
}

void bgpo_trace_reset(bgpo_trace* t) {
  if (t) t->count = 0;
}

int32_t bgpo_trace_count(const bgpo_trace* t) { return t ? t->count : 0; }

bgpo_status bgpo_trace_get(const bgpo_trace* t, int32_t idx, int32_t* kernel_id, float* ms) {
  if (!t || !kernel_id || !ms || idx < 0 || idx >= t->count) return BGPO_ERR_INVALID_ARG;
  if (cudaEventSynchronize(t->stop[idx]) != cudaSuccess ||
      cudaEventElapsedTime(ms, t->start[idx], t->stop[idx]) != cudaSuccess) {
    cudaGetLastError();
    return BGPO_ERR_CUDA;
  }
  *kernel_id = t->ids[idx];
  return BGPO_OK;
}

const char* bgpo_kernel_name(int32_t id) {
  static const char* names[KID_COUNT] = {
      "mask_compact", "gather_rows", "lmhead_fwd_lse", "lse_combine", "seq_reduce",
      "bound_coeffs", "lmhead_dz",   "dx_gemm",        "dx_reduce",   "dw_gemm",
      "group_advantage", "selftest_wait", "vrpo_coeffs", "dz_from_logits", "xm_transpose"};
  return (id >= 0 && id < KID_COUNT) ? names[id] : "?";
}

}  // extern "C"

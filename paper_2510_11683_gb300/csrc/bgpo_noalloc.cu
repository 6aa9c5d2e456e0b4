// bgpo_elbo_fwd_noalloc: the per-sample ELBO forward (masking, compaction,
// gather, LM-head GEMM with online log-sum-exp, per-sequence reduction) run on
// a fixed scratch array compiled into the library, for callers that cannot
// allocate device memory themselves.
//
// Who needs it: host code that owns no device allocator, e.g. a plugin loaded
// into a serving process that plans every byte of device memory up front and
// hands plugins only their input and output buffers, or a caller that must not
// trigger cudaMalloc because it would synchronise the device in the middle of a
// pipelined step. Such a caller cannot provide the workspace that
// bgpo_sample_mask / bgpo_elbo_fwd need.
//
// The scratch is a file-scope __device__ array: every GPU that loads this
// library holds kNoAllocScratchBytes of it until the process exits. Host code
// cannot use the array's name as a device address, so the first call on each
// device looks the address up with cudaGetSymbolAddress (with that device
// current) and caches it together with the id of the CUDA context it belongs
// to; a call that finds another context current (after cudaDeviceReset, for
// instance, the module and its array are loaded again, possibly elsewhere)
// looks it up again. That first call should come before any stream capture.
// All calls share the one array and it keeps the previous call's contents, so
// calls whose GPU work overlaps (two streams, two host threads) race on it.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <mutex>

#include "bgpo.h"
#include "bgpo_internal.h"
#include "bgpo_plan.h"

using namespace bgpo;

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(32) << 20;  // 32 MiB
constexpr int kMaxDevices = 64;

}  // namespace

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

namespace {

std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices];              // device address of g_noalloc_scratch, per device
unsigned long long g_scratch_ctx[kMaxDevices];  // id of the context that address belongs to

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

// Id of the current CUDA context (0 when none is current or it cannot be read).
unsigned long long current_context_id() {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(f);
    else
      cudaGetLastError();
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(f);
    else
      cudaGetLastError();
  });
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (get_current && get_id && get_current(&ctx) == CUDA_SUCCESS && ctx &&
      get_id(ctx, &id) == CUDA_SUCCESS)
    return id;
  return 0;
}

// Device address of the scratch array on the current device, looked up once
// per device and CUDA context.
bgpo_status scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return BGPO_ERR_UNSUPPORTED_DEVICE;
  }
  if (dev < 0 || dev >= kMaxDevices) return BGPO_ERR_UNSUPPORTED_DEVICE;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  const unsigned long long ctx = current_context_id();
  if (!g_scratch_addr[dev] || ctx == 0 || ctx != g_scratch_ctx[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) {
      cudaGetLastError();
      g_scratch_addr[dev] = nullptr;
      return BGPO_ERR_CUDA;
    }
    g_scratch_addr[dev] = p;
    // the lookup makes the device's context current if none was
    g_scratch_ctx[dev] = current_context_id();
  }
  *out = g_scratch_addr[dev];
  return BGPO_OK;
}

bool encode_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                uint64_t pitch_bytes, uint32_t box_inner, uint32_t box_outer) {
  using Fn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                          const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                          CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                          CUtensorMapFloatOOBfill);
  static Fn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<Fn>(f);
    else
      cudaGetLastError();
  });
  if (!fn) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {pitch_bytes};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned_to(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace

extern "C" bgpo_status bgpo_elbo_fwd_noalloc(const bgpo_problem* prob, int32_t j, const void* X,
                                             const void* W, const int32_t* Y, float* t_out,
                                             float* ell_out, void* stream) {
  const bgpo_status st0 = bgpo_validate_problem(prob);
  if (st0 != BGPO_OK) return st0;
  if (j < 0 || j >= prob->n_t) return BGPO_ERR_INVALID_ARG;
  if (!X || !W || !Y || !ell_out) return BGPO_ERR_INVALID_ARG;
  if (!aligned_to(X, 16) || !aligned_to(W, 16) || !aligned_to(Y, 4) || !aligned_to(ell_out, 4) ||
      (t_out && !aligned_to(t_out, 4)) || (prob->resp_len && !aligned_to(prob->resp_len, 4)))
    return BGPO_ERR_ALIGNMENT;
  const Geometry g = make_geometry(prob->B, prob->P, prob->R, prob->H, prob->V);
  // the forward regions of the ordinary workspace layout (the same offsets
  // under every flag); the backward regions do not exist here
  const WsLayout L = make_ws_layout(g, false, false);
  if (L.fwd_bytes > kNoAllocScratchBytes) return BGPO_ERR_WORKSPACE_TOO_SMALL;

  int dev = 0, major = 0, minor = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return BGPO_ERR_UNSUPPORTED_DEVICE;
  }
  if (major != 10 || minor != 3) return BGPO_ERR_UNSUPPORTED_DEVICE;
  void* scratch = nullptr;
  const bgpo_status st1 = scratch_address(&scratch);
  if (st1 != BGPO_OK) return st1;

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const WsPtrs w = ws_pointers(scratch, L, /*forward_only=*/true);
  // The error word (status, where, sample tag, row count) must start at zero;
  // every other region is fully written before it is read within one call.
  if (cudaMemsetAsync(scratch, 0, 64, s) != cudaSuccess) {
    cudaGetLastError();
    return BGPO_ERR_CUDA;
  }
  MaskArgs a;
  a.seed = prob->seed;
  a.b_offset = prob->b_offset;
  a.B = prob->B;
  a.R = prob->R;
  a.j = j;
  a.n_t = prob->n_t;
  a.t_mode = prob->t_mode;
  a.t_out = t_out;
  a.mask_out = nullptr;
  a.resp_len = prob->resp_len;
  CUtensorMap map_xm, map_w;
  if (!encode_map(&map_xm, w.xm, g.H, g.m_pad, g.H * 2, kBK, kBM) ||
      !encode_map(&map_w, W, g.H, g.V, g.H * 2, kBK, kBNHalf))
    return BGPO_ERR_CUDA;
  GemmArgs ga;
  ga.g = g;
  ga.num_pairs = gemm_num_pairs(sms);
  ga.j = j;
  ga.coef = nullptr;
  ga.dW = nullptr;
  if (launch_mask_compact(a, w, s) != cudaSuccess ||
      launch_gather(g, j, X, Y, w, s) != cudaSuccess ||
      launch_gemm(GEMM_FWD, map_xm, map_w, map_xm, ga, w, s) != cudaSuccess ||
      launch_lse_combine(g, j, false, w, s) != cudaSuccess ||
      launch_seq_reduce(g, j, w, ell_out, s) != cudaSuccess)
    return BGPO_ERR_CUDA;
  return BGPO_OK;
}

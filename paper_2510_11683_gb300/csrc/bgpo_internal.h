// Launch interfaces between the C-ABI host code and the kernel translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "bgpo_plan.h"

namespace bgpo {

// Pointers into one workspace (see WsLayout).
struct WsPtrs {
  int32_t* err;
  float* t;
  uint32_t* tnum;    // T numerators as (low, high) 32-bit pairs
  int32_t* seg_off;
  int32_t* rows;
  int32_t* tgt;
  float* tgt_logit;
  float* lse;
  float* logp;
  float2* part;
  void* xm;   // bf16
  void* xmT;  // bf16 [H, dz_rows]
  void* dz;   // bf16 [dz_rows, dz_cols]
  int64_t dz_rows;
  int64_t dz_cols;     // vc (one vocabulary chunk at a time) or v_pad (the whole vocabulary)
  bool dz_chunk_local; // chunk c of dZ starts at column 0 (else at column c vc)
  float* dxp;
  float* zc;  // fp32 logits kept by the forward; null when the layout has none
};

// `forward_only`: the buffer holds only the regions below L.fwd_bytes; the
// backward regions (xmT, dz, dxp, zc) are given as null pointers.
WsPtrs ws_pointers(void* ws, const WsLayout& L, bool forward_only = false);

struct MaskArgs {
  uint64_t seed;
  int32_t b_offset;   // global index of sequence 0 in the Philox counters
  int32_t B, R, j, n_t, t_mode;
  float* t_out;       // may be null
  uint8_t* mask_out;  // may be null
  const int32_t* resp_len;  // may be null: [B] real response lengths
  bool pair_dw = false;     // BGPO_FLAG_PAIR_DW: an odd sample may pair with a pending one
};

cudaError_t launch_mask_compact(const MaskArgs& a, const WsPtrs& w, cudaStream_t s);
cudaError_t launch_gather(const Geometry& g, int32_t j, const void* X, const int32_t* Y,
                          const WsPtrs& w, cudaStream_t s);
// `kept_logits`: the forward GEMM just wrote this sample's logits to w.zc.
cudaError_t launch_lse_combine(const Geometry& g, int32_t j, bool kept_logits, const WsPtrs& w,
                               cudaStream_t s);
// dz of vocabulary chunk `chunk` from the logits the forward kept (same
// arithmetic as the GEMM_DZ epilogue).
cudaError_t launch_dz_from_logits(const Geometry& g, int32_t j, int64_t chunk, const float* coef,
                                  int num_sms, const WsPtrs& w, cudaStream_t s);
cudaError_t launch_seq_reduce(const Geometry& g, int32_t j, const WsPtrs& w, float* ell_out,
                              cudaStream_t s);
cudaError_t launch_bound_coeffs(int32_t B, int32_t n_t, float loss_scale, const float* ell,
                                const float* ell_old, const float* A, float* coef_out,
                                float* g_out, const WsPtrs& w, cudaStream_t s);
cudaError_t launch_dx_reduce(const Geometry& g, int32_t j, const WsPtrs& w, float* dX,
                             cudaStream_t s);
// Xm^T from Xm for the current sample's rows (the dW GEMM reads it K-major),
// from column ERR_ROW_OFF on. `defer`: this sample's dW GEMM waits for the
// next sample's; the kernel records the sample as pending.
cudaError_t launch_xm_transpose(const Geometry& g, int32_t j, bool defer, const WsPtrs& w,
                                cudaStream_t s);
cudaError_t launch_group_advantage(int32_t B, int32_t G, const float* rewards, float* A_out,
                                   cudaStream_t s);
cudaError_t launch_vrpo_coeffs(int32_t B, int32_t n_t, float loss_scale, const float* ell,
                               const float* ell_old, const float* A, float* coef_out, float* R_out,
                               const WsPtrs& w, cudaStream_t s);
cudaError_t launch_selftest_wait(int32_t* err, uint64_t timeout_ns, cudaStream_t s);

// The four tcgen05 GEMMs of the path.
enum GemmKind : int { GEMM_FWD = 0, GEMM_DZ = 1, GEMM_DX = 2, GEMM_DW = 3 };

struct GemmArgs {
  Geometry g;
  int num_pairs;      // CTA pairs launched (gemm_num_pairs)
  int32_t j;
  // GEMM_DZ / GEMM_DX / GEMM_DW: the vocabulary range [v_begin, v_end) of this
  // launch (one chunk of the backward, or the whole vocabulary for a dW GEMM
  // over a whole-vocabulary dZ) and the dZ column where v_begin lies
  int64_t v_begin = 0, v_end = 0, dz_col0 = 0;
  int64_t chunk = 0;  // GEMM_DX: chunk index (chunk 0 stores split partials, later ones add)
  const float* coef;  // GEMM_DZ: per-sequence dL/dl
  float* dW;          // GEMM_DW: accumulated weight gradient [V, H]
  float* dX = nullptr;  // GEMM_DX: accumulated dHidden [B, R, H] (written directly without split-K)
  bool pair_consume = false;  // GEMM_DW: this dW GEMM completes a pair (odd j, BGPO_FLAG_PAIR_DW)
};

// CTA pairs the GEMM kernels run as: the 2-CTA clusters that fit on the
// device at once (at most num_sms / 2), so that every pair of the persistent
// grid is resident.
int gemm_num_pairs(int num_sms);

// map_a / map_b: the operand tiles; map_c: the epilogue's destination (the
// fp32 logit region for GEMM_FWD when w.zc is set, dZ for GEMM_DZ, the split-K
// partials for GEMM_DX, dW for GEMM_DW).
cudaError_t launch_gemm(GemmKind kind, const CUtensorMap& map_a, const CUtensorMap& map_b,
                        const CUtensorMap& map_c, const GemmArgs& a, const WsPtrs& w,
                        cudaStream_t s);

}  // namespace bgpo

/*
 * bgpo.h -- C ABI of the GB300 (sm_103a) BGPO masked-diffusion ELBO hot path.
 *
 * Boundary-Guided Policy Optimization (arxiv 2510.11683) trains a diffusion LLM
 * on a linear lower bound of its ELBO-based RL objective. Per Monte Carlo sample
 * j of each response b the path is:
 *
 *   bgpo_sample_mask          t_{b,j} and the response mask (Sec. 2.1; Eq. 3, 5;
 *                             Algorithm 1, sampling of t and y_t)
 *   bgpo_elbo_fwd             l_{b,j} = (1/t) sum_masked log p(y^i | y_t, x) through
 *                             the LM head (Eq. 4), full logits never stored
 *   bgpo_bound_coeffs         d_j (Eq. 10), g_j (Eq. 13) and dL_j/dl_j with
 *                             L_j = -loss_scale * g_j (Algorithm 1; Eq. 19)
 *   bgpo_elbo_bwd_accumulate  dX += dL_j/dX, dW += dL_j/dW (Algorithm 1, gradient
 *                             accumulation; Linearity, Sec. 3), so memory does
 *                             not grow with n_t
 *
 * plus bgpo_group_advantage (Eq. 18) and, for comparison, the coefficients of
 * the ELBO-based objective the bound replaces (bgpo_vrpo_coeffs, Eq. 7).
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Pointers marked "device" are CUDA device pointers on the current device;
 *    "host" pointers are ordinary host memory. The caller allocates and owns
 *    every buffer, including one workspace of bgpo_workspace_bytes() bytes.
 *    The library allocates no device memory.
 *  - All launches are asynchronous on `stream` (a cudaStream_t; NULL = the
 *    legacy default stream). No call synchronises except
 *    bgpo_get_device_error and bgpo_trace_get.
 *  - Dtypes are fixed: X and W bfloat16, Y int32, everything else float32.
 *  - Layouts are dense row-major: X [B, P+R, H], W [V, H], Y [B, R],
 *    dX [B, R, H] (response rows only), dW [V, H], per-sequence vectors [B].
 *  - Alignment: X, W, dX, dW and the workspace must be 16-byte aligned
 *    (workspace: 256-byte). H must be a multiple of 8 (16-byte rows of X and W).
 *  - The workspace carries sample j's draws (t, mask), its compacted masked
 *    rows, forward statistics and (with BGPO_FLAG_KEEP_LOGITS) the masked
 *    rows' logits from one call to the next, so the calls for
 *    one sample must be issued in the order
 *        bgpo_sample_mask -> bgpo_elbo_fwd -> [bgpo_bound_coeffs] ->
 *        bgpo_elbo_bwd_accumulate
 *    on one stream, with the same j. A call made with a j other than the one
 *    the workspace holds sets the device error word to BGPO_ERR_INVALID_ARG
 *    and does no work. With BGPO_FLAG_PAIR_DW the workspace also carries an
 *    even sample's dL/dz rows into the next sample's backward (see the flag).
 *  - Host-side checks return a status before anything is launched. A failed
 *    launch returns BGPO_ERR_CUDA. Faults detected on the device (a non-finite
 *    coefficient, a bounded wait that ran out, a sample mismatch) are recorded
 *    in an error word inside the workspace: read it with bgpo_get_device_error.
 *  - The device must have compute capability 10.3 (GB300); otherwise every
 *    launching call returns BGPO_ERR_UNSUPPORTED_DEVICE.
 *  - A checked build of the same library (compiled with -DBGPO_CHECKED) tests
 *    every index it reads from device memory (masked-row lists, segment
 *    offsets, row counts, split counts) and every target token against its
 *    buffer before use; a failed test records BGPO_ERR_BOUNDS in the error word
 *    and skips the access. It stands in for a memory checker. The normal build
 *    trusts these values, which its own kernels wrote.
 */
#ifndef BGPO_H_
#define BGPO_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BGPO_ABI_VERSION 3

typedef enum bgpo_status {
  BGPO_OK = 0,
  BGPO_ERR_INVALID_ARG = 1,          /* null pointer, j out of range, bad enum */
  BGPO_ERR_SHAPE = 2,                /* sizes out of the supported range */
  BGPO_ERR_ALIGNMENT = 3,            /* pointer not aligned as required */
  BGPO_ERR_WORKSPACE_TOO_SMALL = 4,  /* ws_bytes < bgpo_workspace_bytes() */
  BGPO_ERR_NONFINITE = 5,            /* non-finite bound coefficient (device) */
  BGPO_ERR_UNSUPPORTED_DEVICE = 6,   /* current device is not sm_103 */
  BGPO_ERR_CUDA = 7,                 /* a CUDA runtime call or launch failed */
  BGPO_ERR_TIMEOUT = 8,              /* a bounded device-side wait ran out */
  BGPO_ERR_BOUNDS = 9                /* checked build only: an index read from device
                                        memory fell outside its buffer; the access
                                        was skipped (device) */
} bgpo_status;

/* Optional per-kernel timing: CUDA events recorded around each kernel launch. */
typedef struct bgpo_trace bgpo_trace;

/* t_mode values */
#define BGPO_T_IID 0         /* t_{b,j} i.i.d. on (0, 1] (Eq. 5) */
#define BGPO_T_STRATIFIED 1  /* t_{b,j} in (j/n_t, (j+1)/n_t]; not in the paper */

/*
 * flags bits
 *   BGPO_FLAG_KEEP_LOGITS  bgpo_elbo_fwd also writes the fp32 logits z = Xm W^T
 *       of the masked rows into the workspace, and the backward of that sample
 *       forms dL/dz from them in one HBM-bound pass instead of recomputing the
 *       logits with a fourth tensor-core GEMM. Same results bit for bit, a
 *       quarter less tensor-core work per sample, and
 *       4 * roundup(B R, 256) * roundup(V, 64) more workspace bytes. Without
 *       it (the default) full logits never reach device memory. Leave it off
 *       for forward-only passes (the old policy's l_old).
 */
#define BGPO_FLAG_KEEP_LOGITS 1u
/*
 *   BGPO_FLAG_PAIR_DW  consecutive MC samples (2k, 2k + 1) share one dW GEMM
 *       whose K range holds both samples' masked rows (M_2k + M_2k+1 instead
 *       of M_j), so dW's fp32 read-modify-write (8 V H bytes) happens once per
 *       pair instead of once per sample. The backward of an even sample j < n_t - 1
 *       updates dX as usual but leaves its dL/dz rows and gathered hidden
 *       states pending in the workspace and adds nothing to dW; the backward of
 *       sample j + 1 on the same workspace adds both samples' dW contributions.
 *       dW is therefore complete after the backward of every odd sample and of
 *       the last sample (j = n_t - 1), i.e. at the end of Algorithm 1's loop,
 *       but not between the two backward calls of a pair. The same dW up to
 *       fp32 summation order; dX and l are unchanged bit for bit. The dZ and
 *       Xm^T regions of the workspace double: 2 * roundup(B R, 256) *
 *       (roundup(V, 64) + H) more bytes, independent of n_t. Every call on
 *       the workspace within a step must carry the flag. Misuse is reported in
 *       the device error word as BGPO_ERR_INVALID_ARG: the backward of an odd
 *       sample whose partner is not pending (its dW then holds sample j
 *       alone), or the masking of another sample while one is pending (the
 *       pending contribution is dropped). bgpo_clear_device_error forgets a
 *       pending sample. A repeated backward of the same odd sample adds that
 *       sample's dW alone, as without the flag. Keeping every sample's
 *       workspace apart (bgpo_vrpo_coeffs' "retain" strategy) does not pair:
 *       leave the flag off there.
 */
#define BGPO_FLAG_PAIR_DW 2u

/*
 * Problem description (host struct, read by every call; never stored).
 *   B      responses in the batch (>= 1)
 *   P      prompt length: X rows [b, 0, P) are the prompt, never masked (Sec. 2.1)
 *   R      response length (>= 1); response position i is X row [b, P + i]
 *   H      hidden size, multiple of 8, 64 <= H <= 16384 (a last K block or hidden-size
 *          tile that H does not fill is read as zeros and written only up to H)
 *   V      vocabulary size, 1 <= V <= 2^24
 *   n_t    MC samples per response, 1 <= n_t < 65536 (Eq. 5)
 *   G      group size used by bgpo_group_advantage (Eq. 18), >= 1
 *   t_mode BGPO_T_IID or BGPO_T_STRATIFIED
 *   seed   Philox4x64-10 key word 0; the draws of (b, j) depend on (seed, b_offset + b, j)
 *   loss_scale  L_j = -loss_scale * g_j; Algorithm 1 uses 1/G
 *   b_offset  global index of this batch's first sequence (>= 0). A data-parallel
 *          shard holding sequences [b_offset, b_offset + B) of a larger batch
 *          draws exactly the t and masks the whole batch would draw for them.
 *   trace  optional bgpo_trace* (NULL = off)
 *   resp_len  optional device int32 [B] (NULL = every response has R tokens):
 *          response b holds resp_len[b] tokens (0 <= resp_len[b] <= R); positions
 *          i >= resp_len[b] are padding and never masked (the draws of the other
 *          positions are unchanged; values outside [0, R] are clamped)
 *   flags  BGPO_FLAG_* bits (0 = defaults); other bits are rejected
 *   vocab_chunk  columns of the vocabulary the backward handles at a time
 *          (0 = default, else a positive multiple of 256; BGPO_ERR_INVALID_ARG
 *          otherwise). The backward forms dL/dz, its dX contribution and its
 *          dW rows one chunk of the vocabulary after another, so the dL/dz
 *          buffer in the workspace holds roundup(B R, 256) x vocab_chunk
 *          bf16 values instead of roundup(B R, 256) x V (Linearity, Sec. 3: the
 *          gradient is a sum over vocabulary entries as well as over samples).
 *          Default: the whole vocabulary at once when its dL/dz takes at most
 *          1 GiB (2 roundup(B R, 256) roundup(V, 64) bytes) or with
 *          BGPO_FLAG_PAIR_DW (whose even samples leave their dL/dz for the
 *          whole vocabulary pending); otherwise chunks of at most 32768
 *          columns (V split evenly, rounded up to 256). A chunk of V or more
 *          columns is the whole vocabulary at once. l and dW are the same
 *          bits for every chunk width; dX is the same sum up to fp32 order.
 * B * R must not exceed 2^22 and B * R * V must fit the workspace (see
 * bgpo_workspace_bytes).
 */
typedef struct bgpo_problem {
  int32_t B;
  int32_t P;
  int32_t R;
  int32_t H;
  int32_t V;
  int32_t n_t;
  int32_t G;
  int32_t t_mode;
  uint64_t seed;
  float loss_scale;
  int32_t b_offset;
  bgpo_trace* trace;
  const int32_t* resp_len;
  uint32_t flags;
  int32_t vocab_chunk;
} bgpo_problem;

/* ABI version of the loaded library (BGPO_ABI_VERSION). */
int32_t bgpo_abi_version(void);

/* Human-readable name of a status code (static string). */
const char* bgpo_status_string(bgpo_status status);

/*
 * Host-only validation of a problem description (no CUDA call).
 * Returns BGPO_OK, BGPO_ERR_INVALID_ARG (NULL, bad t_mode, negative b_offset,
 * non-finite loss_scale, unknown flags, vocab_chunk negative or not a multiple
 * of 256) or BGPO_ERR_SHAPE.
 */
bgpo_status bgpo_validate_problem(const bgpo_problem* prob);

/*
 * Bytes of device workspace the calls below need for `prob`. Depends on B, R,
 * H, V, the flags and vocab_chunk only -- never on n_t (Linearity, Sec. 3: one
 * sample's state at a time; with BGPO_FLAG_PAIR_DW two). A workspace sized with
 * a flag also serves calls made without it and the same vocab_chunk. Returns 0
 * for an invalid problem.
 */
size_t bgpo_workspace_bytes(const bgpo_problem* prob);

/*
 * Forward masking process for MC sample j (Sec. 2.1; Eq. 3, 5; Algorithm 1).
 * Draws t_{b,j} = T/D with Philox4x64-10 (key (seed, 0), counter (0, b', j, 1)
 * with b' = b_offset + b the global sequence index,
 * T = u24 + 1 and D = 2^24, or T = j 2^24 + u24 + 1 and D = n_t 2^24 when
 * stratified; u24 = top 24 bits of output word 0) and masks response position
 * i of sequence b iff u24_i * D < T * 2^24, where u24_i is the top 24 bits of
 * output word (i mod 4) of the block with counter (i / 4, b', j, 0). Prompt
 * positions, and response positions at or past resp_len[b], are never masked.
 * Compacts the masked positions into ascending
 * (b, i) order inside the workspace.
 *   j         sample index, 0 <= j < n_t
 *   ws        device workspace (256-byte aligned), ws_bytes its size
 *   t_out     device float [B] or NULL: t_{b,j} rounded to float
 *   mask_out  device uint8 [B, R] or NULL: 1 = masked
 */
bgpo_status bgpo_sample_mask(const bgpo_problem* prob, int32_t j, void* ws, size_t ws_bytes,
                             float* t_out, uint8_t* mask_out, void* stream);

/*
 * Per-step ELBO term of Eq. 4 for sample j, every sequence:
 *   l_{b,j} = (1 / t_{b,j}) * sum_{i masked} log softmax(W x_{b,P+i})[Y[b,i]]
 * (no length normalisation; an empty mask gives 0). The masked rows of X are
 * gathered, multiplied by W on the tensor cores (bf16 in, fp32 accumulate)
 * and reduced by an online log-sum-exp per row; the per-row log-sum-exp and
 * log-probabilities stay in the workspace for the backward pass. Full logits
 * are never written, unless BGPO_FLAG_KEEP_LOGITS asks for the masked rows'
 * fp32 logits to stay in the workspace. The result is
 * deterministic (fixed reduction order), so recomputing l with unchanged inputs
 * gives bit-identical values (on-policy d_j = 0 exactly, Sec. 3.2).
 *   X      device bf16 [B, P+R, H];  W device bf16 [V, H];  Y device int32 [B, R]
 *          with 0 <= Y < V (out-of-range targets give an undefined l)
 *   ell_out device float [B]: l_{b,j} (e.g. column j of a [n_t, B] array)
 * Requires a preceding bgpo_sample_mask(j) on the same workspace.
 */
bgpo_status bgpo_elbo_fwd(const bgpo_problem* prob, int32_t j, const void* X, const void* W,
                          const int32_t* Y, void* ws, size_t ws_bytes, float* ell_out,
                          void* stream);

/*
 * BGPO bound coefficients for sample j (Eq. 10, 13; Algorithm 1; Eq. 19):
 *   d     = ell - ell_old                       (same t and mask for both policies)
 *   g     = (1 + d) A / n_t        if A >= 0    (Lemma 1, Taylor)
 *           e^d A / n_t            if A <  0    (Lemma 2, Jensen)
 *   coef  = dL_j / dl_j = -loss_scale * A * (A >= 0 ? 1 : e^d) / n_t
 * All pointers device float [B]. g_out may be NULL. A non-finite g or coef
 * sets the device error word to BGPO_ERR_NONFINITE (values are still written).
 */
bgpo_status bgpo_bound_coeffs(const bgpo_problem* prob, int32_t j, const float* ell,
                              const float* ell_old, const float* A, float* coef_out, float* g_out,
                              void* ws, size_t ws_bytes, void* stream);

/*
 * Coefficients of the ELBO-based objective BGPO bounds (VRPO, Eq. 7), for
 * comparison with the bound: with B_hat the mean over the n_t samples (Eq. 5),
 *   R_hat = e^{mean_j (l_{b,j} - l_old_{b,j})} A_b
 *   coef  = dL/dl_{b,j} = -loss_scale * A_b * e^{mean_j d_{b,j}} / n_t  (every j)
 * Unlike bgpo_bound_coeffs it needs all n_t samples' l before any backward
 * pass: the caller either keeps every sample's workspace (memory grows with
 * n_t) or runs each sample's forward twice. Feed coef to
 * bgpo_elbo_bwd_accumulate for each j. On-policy (d = 0) it equals the
 * bound's coefficient (Equivalence, Sec. 3.2).
 *   ell, ell_old  device float [n_t, B] (row j = sample j);  A device float [B]
 *   coef_out      device float [B];  R_out device float [B] or NULL
 * A non-finite value sets the device error word to BGPO_ERR_NONFINITE.
 */
bgpo_status bgpo_vrpo_coeffs(const bgpo_problem* prob, const float* ell, const float* ell_old,
                             const float* A, float* coef_out, float* R_out, void* ws,
                             size_t ws_bytes, void* stream);

/*
 * Backward pass of L_j = sum_b coef_b * l_{b,j}, accumulated (Algorithm 1,
 * gradient accumulation; Eq. 15-17 give the per-sample gradient weights):
 *   w_r   = coef_b / t_{b,j}                       for masked row r = (b, i)
 *   dz_r  = w_r (onehot(Y[b,i]) - softmax(W x_r))  (bf16; logits recomputed
 *           on the tensor cores, or with BGPO_FLAG_KEEP_LOGITS read from what
 *           bgpo_elbo_fwd kept; the two give identical bits)
 *   dX[b, i, :] += W^T dz_r        dW += sum_r dz_r x_r^T
 * computed one vocabulary chunk at a time (see bgpo_problem.vocab_chunk):
 * dz of the chunk, then its terms of dX and of the chunk's rows of dW.
 * Per-sample hidden states: in the paper p_theta conditions on the masked
 * sequence (Sec. 2.1), so each MC sample may have its own X. Pass sample j's
 * X_j to bgpo_elbo_fwd and to this call: dX then receives dL_j/dX_j, the
 * gradient of sample j's own hidden states, added to what dX holds (zero it
 * before each sample to read it per sample), and dW accumulates over samples.
 * Under BGPO_FLAG_PAIR_DW the pending even sample's gathered hidden states
 * (taken from its own X_j) stay in the workspace for the pair's dW GEMM.
 * (with BGPO_FLAG_PAIR_DW the dW term of an even sample is added by the next
 * sample's call.)
 * coef is an input (normally bgpo_bound_coeffs' output for the same j).
 *   dX device float [B, R, H], dW device float [V, H]: accumulated in place.
 * Deterministic: no atomics, fixed summation order.
 * Requires bgpo_sample_mask(j) and bgpo_elbo_fwd(j) before it on the same
 * workspace, with the same X, W and Y. With BGPO_FLAG_KEEP_LOGITS the last
 * bgpo_elbo_fwd of sample j must have kept its logits (been called with the
 * flag too); otherwise the device error word is set to BGPO_ERR_INVALID_ARG
 * and dX and dW are left unchanged.
 */
bgpo_status bgpo_elbo_bwd_accumulate(const bgpo_problem* prob, int32_t j, const void* X,
                                     const void* W, const int32_t* Y, const float* coef, void* ws,
                                     size_t ws_bytes, float* dX, float* dW, void* stream);

/*
 * Group-normalised advantages (Eq. 18) over consecutive groups of G responses:
 *   A = (r - mean_G r) / std_G r, population std; a zero-std group gets A = 0.
 *   rewards, A_out: device float [B]; B must be a multiple of G.
 */
bgpo_status bgpo_group_advantage(const bgpo_problem* prob, const float* rewards, float* A_out,
                                 void* stream);

/*
 * bgpo_elbo_fwd_noalloc -- bgpo_sample_mask(j) followed by bgpo_elbo_fwd(j)
 * with no caller-provided workspace: the scratch lives in a fixed array
 * compiled into the library. The paper has no counterpart; this entry point
 * exists for callers that cannot allocate device memory -- host code given
 * only its input and output buffers by a process that plans all device
 * memory itself, or code that must not call cudaMalloc because it would
 * synchronise the device -- and so cannot pass the workspace the other calls
 * need.
 *   X, W, Y   as for bgpo_elbo_fwd;  t_out device float [B] or NULL;
 *   ell_out   device float [B]: l_{b,j} (Eq. 4), same values as bgpo_elbo_fwd.
 * It keeps no logits (prob->flags is validated, then ignored). prob->resp_len,
 * when given, must be 4-byte aligned like the other int32 pointers
 * (BGPO_ERR_ALIGNMENT otherwise, before anything is launched).
 * Limit: the forward scratch of `prob` must fit the 32 MiB array, about
 * roundup(B*R, 256) * (2 H + 8 ceil(V / 256) + 20) + 16 B + 12288 bytes;
 * larger problems return BGPO_ERR_WORKSPACE_TOO_SMALL before anything is
 * launched. Every GPU that loads the library holds the 32 MiB until the
 * process exits. The first call on each device looks up the array's device
 * address (cudaGetSymbolAddress, with that device current) and caches it with
 * the id of the current CUDA context; a call that finds another context
 * current (after cudaDeviceReset, say) looks it up again. That first call
 * should come before any stream capture. Calls allocate nothing and free
 * nothing.
 * All calls share the one array, which keeps the previous call's contents:
 * calls whose GPU work overlaps (other streams, other host threads) race and
 * give undefined results. Device-side errors are recorded in the array's own
 * error word, which the next call clears; use bgpo_elbo_fwd with a workspace
 * to read them.
 */
bgpo_status bgpo_elbo_fwd_noalloc(const bgpo_problem* prob, int32_t j, const void* X,
                                  const void* W, const int32_t* Y, float* t_out, float* ell_out,
                                  void* stream);

/*
 * Reads the device error word of a workspace (synchronises `stream`).
 *   code_out: BGPO_OK or the first device-detected status; where_out (may be
 *   NULL): kernel and site that set it.
 */
bgpo_status bgpo_get_device_error(const void* ws, size_t ws_bytes, int32_t* code_out,
                                  int32_t* where_out, void* stream);

/* Clears the device error word (asynchronous on `stream`) and forgets a
 * sample pending under BGPO_FLAG_PAIR_DW. Clear a new workspace before its
 * first call. */
bgpo_status bgpo_clear_device_error(void* ws, size_t ws_bytes, void* stream);

/*
 * Failure-detection self-test: one warp waits, with the bounded wait every
 * kernel of this library uses, on a barrier that nothing arrives at. After
 * timeout_us (1 .. 1,000,000) the wait gives up and the kernel records
 * BGPO_ERR_TIMEOUT in the workspace's device error word; the CUDA context stays
 * usable. ws: a workspace (only its error word is touched).
 */
bgpo_status bgpo_selftest_bounded_wait(void* ws, size_t ws_bytes, uint32_t timeout_us,
                                       void* stream);

/* ---- per-kernel timing (host objects holding CUDA events) ---------------- */

/* Creates a trace that can hold `capacity` kernel launches; NULL on failure.
 * A trace records from one host thread at a time: calls that may run
 * concurrently need their own traces. */
bgpo_trace* bgpo_trace_create(int32_t capacity);
void bgpo_trace_destroy(bgpo_trace* trace);
/* Forgets recorded launches (events are reused). */
void bgpo_trace_reset(bgpo_trace* trace);
int32_t bgpo_trace_count(const bgpo_trace* trace);
/* Kernel id and duration in ms of recorded launch idx (waits for it). */
bgpo_status bgpo_trace_get(const bgpo_trace* trace, int32_t idx, int32_t* kernel_id, float* ms);
/* Name of a kernel id (static string), "?" if unknown. */
const char* bgpo_kernel_name(int32_t kernel_id);

#ifdef __cplusplus
}
#endif

#endif /* BGPO_H_ */

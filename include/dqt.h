/*
 * dqt.h -- C ABI of the GB300 (sm_103a) Direct Quantized Training library.
 *
 * Direct Quantized Training (DQT; Zhao et al., "Direct Quantized Training of
 * Language Models with Stochastic Rounding", arXiv 2412.04787) trains
 * BitLinear layers whose weights exist only as n-bit integer codes c with a
 * fixed per-tensor scale s_w (W_tilde = c / s_w, Eq. 2-4).  One training step
 * of a layer is:
 *
 *   dqt_act_quant                 8-bit per-token absmax activation codes (Sec. 3.2)
 *   dqt_bitlinear_fwd             Y = X_tilde W_tilde^T, exact integer accumulation (Sec. 3.2)
 *   dqt_bitlinear_bwd_dx          dX = dY W_tilde (Sec. 3.2; no STE on the weight)
 *   dqt_bitlinear_bwd_dw_update   dW = dY^T X_tilde, then in the GEMM epilogue the AdamW
 *                                 step (Sec. 4.1) and W_hat = SR(W') (Eq. 1, Eq. 5),
 *                                 clamped to the n-bit grid and written over the codes
 *   dqt_sr_update                 the same AdamW + SR step for a gradient given in memory
 *                                 (dqt_sr_t.elem0: a data-parallel shard's global offset)
 *   dqt_*_fp8                     the forward with E4M3 operands (FP8 environment, Sec. 4.3)
 *   dqt_*packed*                  2-bit packed ternary code storage (Sec. 1)
 *   dqt_*adafactor*               Adafactor with SR instead of AdamW (Sec. 4.3)
 *
 * and, not part of the method, four operations of the LLaMA-structured decoder
 * (the model family of Sec. 4.1) built around those layers: dqt_rope_bf16,
 * dqt_swiglu_bf16 / dqt_swiglu_bwd_bf16, dqt_rmsnorm_bf16 / dqt_rmsnorm_bwd_bf16,
 * dqt_cross_entropy_fwd_bf16 / _bwd_bf16.
 *
 * GB300 has no int8 tensor-core MMA for sm_103a, so the integer GEMMs run on
 * the bf16 tensor cores over exact bf16 images of the integer codes (every
 * integer in [-256, 256] is exact in bf16; products and partial sums below
 * 2^24 are exact in the fp32 accumulator).  The hot-path
 * calls take the int8 codes themselves and make the bf16 operands they need
 * in a caller-provided workspace (dqt_codes_to_bf16, dqt_codes_to_xdq) before
 * the GEMM.  The *_img calls take those images directly
 * (dqt_act_quant_images, dqt_codes_to_bf16) for callers that share one image
 * between several GEMMs.
 *
 * Conventions for every entry point:
 *   - All data pointers are DEVICE pointers owned by the caller; the library
 *     keeps no reference after the call returns and allocates no device memory.
 *   - Every call is asynchronous on `stream` (a cudaStream_t; NULL selects the
 *     legacy default stream).  Host-side argument checks run before any launch;
 *     a non-zero return means nothing was launched (except DQT_ERR_CUDA, which
 *     reports a launch failure).
 *   - bf16 tensors are passed as dqt_bf16 (the raw IEEE bfloat16 bits).
 *   - Matrices are row-major and contiguous.  Device pointers must be 16-byte
 *     aligned and the row lengths K and N multiples of 8 (the tensor-memory
 *     accelerator moves 16-byte rows); otherwise DQT_ERR_ALIGN.
 *   - Device-side waits are bounded.  A kernel whose wait runs out records
 *     DQT_ERR_TIMEOUT in a device status word and returns early, leaving its
 *     outputs undefined; dqt_check_device_status() reports and clears it.
 */
#ifndef DQT_H_
#define DQT_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t dqt_bf16; /* raw bfloat16 bits */

enum {
  DQT_OK = 0,
  DQT_ERR_ARG = 1,     /* null pointer, bad size, bad grid or hyper-parameter   */
  DQT_ERR_ALIGN = 2,   /* pointer not 16-byte aligned, K or N not a multiple of 8 */
  DQT_ERR_CUDA = 3,    /* a CUDA runtime or driver call failed                   */
  DQT_ERR_TIMEOUT = 4, /* a bounded device wait ran out (dqt_check_device_status) */
  DQT_ERR_RANGE = 5    /* a size exceeds what the kernels index (see each call)  */
};

/* The n-bit grid [Q_n, Q_p] of Eq. 3.  Ternary ("1.58-bit") is [-1, 1]; an
 * integer width n in [2, 8] is [-2^(n-1), 2^(n-1) - 1].  Codes are int8. */
typedef struct {
  int32_t qmin;
  int32_t qmax;
} dqt_grid_t;

/* AdamW hyper-parameters (the optimiser of Sec. 4.1).  step >= 1 is the
 * 1-based optimiser step used for the bias corrections bc1 = 1 - beta1^step,
 * bc2 = 1 - beta2^step; eps > 0.  The library derives, in fp64 rounded once
 * to fp32: 1 - beta1, 1 - beta2, k1 = bc1 / sqrt(bc2), k2 = bc1 * eps,
 * 1 - lr * weight_decay and lr * s_w, and evaluates AdamW's
 * m_hat / (sqrt(v_hat) + eps) as m / (sqrt(v) * k1 + k2). */
typedef struct {
  float lr;
  float beta1;
  float beta2;
  float eps;
  float weight_decay;
  int64_t step;
} dqt_adamw_t;

/* Stochastic rounding stream (Eq. 1).  The uniform for element e (global
 * flat row-major index into the weight tensor) is word e % 4 of
 * Philox4x32-10(counter = (e/4 low 32, e/4 high 32, step low 32, tensor_id),
 * key = (seed low 32, seed high 32)), U = (word >> 8) * 2^-24; the code rounds
 * up when U < x - floor(x).  round_mode 0 = stochastic rounding (the paper's
 * method); 1 = round to nearest (the absmax-without-SR ablation of Sec. 5.1).
 * elem0: the global index of the first element a call updates (element i of
 * the call is global element elem0 + i; for a weight-gradient call, element
 * (n, k) is elem0 + n K + k).  0 for a whole tensor; a data-parallel rank
 * that updates the shard [a, b) of a flat weight passes elem0 = a, so the
 * codes do not depend on how the tensor is sharded.  elem0 >= 0 and a
 * multiple of 4 (one Philox block per four elements), else DQT_ERR_ARG /
 * DQT_ERR_ALIGN.  The Adafactor calls need elem0 = 0 (their factored
 * statistics span the whole matrix). */
typedef struct {
  uint64_t seed;
  uint32_t tensor_id;
  int32_t round_mode;
  int64_t elem0;
} dqt_sr_t;

/* Eq. 3: grid for `bits` in {1.58, 2, 3, ..., 8}.  Host only. */
int dqt_grid_for_bits(float bits, dqt_grid_t* out);

/* Human-readable name of a status code.  Host only; never NULL. */
const char* dqt_status_string(int status);

/* Synchronises `stream`, then returns DQT_ERR_TIMEOUT if any kernel of this
 * library recorded a timed-out wait since the last call (and clears the
 * record), DQT_ERR_CUDA if the stream reports an error, else DQT_OK. */
int dqt_check_device_status(void* stream);

/* Upper bound, in nanoseconds, on any single device-side wait of this
 * library's kernels (default 2e9).  Applies to launches made after the call. */
int dqt_set_wait_limit_ns(uint64_t ns);

/* GEMM tiling for launches made after the call (host setting, all devices):
 * 0 (default) = 2-SM tiles: a cluster of two CTAs on one TPC computes a
 *     256 x 256 tile with tcgen05.mma.cta_group::2;
 * 1 = 1-SM 128 x 256 tiles.
 * Forward GEMMs whose exact integer accumulation needs fp32 chunks drained
 * into int32 (codes wider than 4 bits with K > 1024) always use 1-SM tiles.
 * Results are identical either way (the same per-element arithmetic);
 * DQT_ERR_ARG for any other mode. */
int dqt_set_gemm_tiles(int mode);

/* Eq. 2-4, initialisation (not on the training hot path).
 *   W0      fp32 [numel] dense initial weight (device)
 *   codes   int8 [numel] out: Clip[Round(W0 * s_w), qmin, qmax], Round half-to-even
 *   s_w     HOST float out: qmax / AbsMean(W0), AbsMean = (1/numel) sum |w| in fp64
 *   ws      device workspace of at least dqt_absmean_workspace_size() bytes
 * Synchronous: returns after s_w is known and the codes kernel is enqueued. */
size_t dqt_absmean_workspace_size(void);
int dqt_absmean_init(const float* W0, int64_t numel, dqt_grid_t grid, int8_t* codes,
                     float* s_w, void* ws, size_t ws_bytes, void* stream);

/* The AbsMean initialisation of dqt_absmean_init for callers that cannot
 * allocate device memory (a framework that owns every device allocation
 * through its own pool, code inside an allocator's own set-up, a job whose
 * memory budget is fully reserved).  The paper has no counterpart: this is a
 * deployment variant only.  It takes no workspace: the reduction's partial
 * sums live in a static device array of 1025 doubles (8200 bytes) that every
 * GPU loading the library holds until the process exits.  Same arguments and
 * results as dqt_absmean_init; numel <= 2^53, else DQT_ERR_RANGE.  It calls
 * no allocator.  Each call looks up (and caches) the array's device address
 * on the current device.  All calls on a device share the array: calls that
 * overlap on the GPU race, so serialise them.  Synchronous, like
 * dqt_absmean_init: every call waits for `stream` and copies the mean to the
 * host, so it must not be called on a stream that is being captured. */
int dqt_absmean_init_noalloc(const float* W0, int64_t numel, dqt_grid_t grid, int8_t* codes,
                             float* s_w, void* stream);

/* Sec. 3.2, activation quantisation "following BitNet", 8 bits per token:
 *   amax[t] = max_k |X[t,k]|,  s_x[t] = 127 / max(amax[t], 1e-5)   (fp32 divide)
 *   Xq[t,k] = Clip[Round(X[t,k] * s_x[t]), -128, 127]              (fp32 multiply, half-to-even)
 *   X       bf16 [T, K] in (16-byte aligned, K a multiple of 8)
 *   Xq      int8 [T, K] out (8-byte aligned)
 *   s_x     fp32 [T] out
 * One pass: 2 bytes read and 1 byte written per element, 4 bytes per row. */
int dqt_act_quant(const dqt_bf16* X, int64_t T, int64_t K, int8_t* Xq, float* s_x,
                  void* stream);

/* dqt_act_quant that can also write the 16-bit GEMM operand images in the
 * same pass (for the *_img calls):
 *   Xq      int8 [T, K] out, or NULL
 *   Xq_img  bf16 [T, K] out, or NULL: the codes as exact bf16 values (forward operand)
 *   Xdq     bf16 [T, K] out, or NULL: bf16(Xq / s_x), the dequantised activation
 *           X_tilde that the weight gradient uses (weight-gradient operand)
 * At least one of Xq, Xq_img, Xdq must be non-NULL; s_x is required. */
int dqt_act_quant_images(const dqt_bf16* X, int64_t T, int64_t K, int8_t* Xq, float* s_x,
                         dqt_bf16* Xq_img, dqt_bf16* Xdq, void* stream);

/* Exact bf16 image of int8 codes: W_img[i] = (bf16) W[i].  numel >= 1.
 * (dqt_bitlinear_bwd_dx runs this into its workspace.) */
int dqt_codes_to_bf16(const int8_t* W, int64_t numel, dqt_bf16* W_img, void* stream);

/* The dequantised activation image from int8 codes: Xdq[t,k] = bf16(Xq[t,k] /
 * s_x[t]) (correctly rounded fp32 division, then bf16), bit-identical to the
 * Xdq of dqt_act_quant_images.  (dqt_bitlinear_bwd_dw_update runs this into
 * its workspace.)  Xq int8 [T, K], s_x fp32 [T], Xdq bf16 [T, K]; K a multiple
 * of 16; Xq, Xdq 16-byte aligned. */
int dqt_codes_to_xdq(const int8_t* Xq, const float* s_x, int64_t T, int64_t K, dqt_bf16* Xdq,
                     void* stream);

/* Sec. 3.2 forward, Y = X_tilde W_tilde^T with X_tilde = Xq / s_x, W_tilde = c / s_w:
 *   acc[t,n] = sum_k Xq[t,k] c[n,k]             exact (int32)
 *   Y[t,n]   = bf16( float(acc) * (1 / (s_x[t] * s_w)) )
 *   Xq       int8 [T, K] activation codes from dqt_act_quant
 *   s_x      fp32 [T]
 *   W        int8 [N, K] weight codes c
 *   grid     the weight grid; it bounds |c| and so how often the kernel drains its
 *            fp32 accumulator into int32 to keep every partial sum exact
 *   Y        bf16 [T, N] out;  acc_out int32 [T, N] out, or NULL
 *   ws       device workspace of at least dqt_fwd_workspace_size(T, K, N) bytes
 *            (16-byte aligned): it receives the exact bf16 images of Xq and W
 *            (3 bytes moved per element of each), which the GEMM then reads,
 *            and the partials of the last-wave slices (dqt_bitlinear_fwd_img)
 * K, N multiples of 8; Xq, W, Y, acc_out 16-byte aligned; T >= 1; T, N, K < 2^31. */
size_t dqt_fwd_workspace_size(int64_t T, int64_t K, int64_t N);
int dqt_bitlinear_fwd(const int8_t* Xq, const float* s_x, const int8_t* W, float s_w,
                      dqt_grid_t grid, int64_t T, int64_t K, int64_t N, dqt_bf16* Y,
                      int32_t* acc_out, void* ws, size_t ws_bytes, void* stream);

/* The same forward on the bf16 operand images (dqt_act_quant_images' Xq_img
 * and dqt_codes_to_bf16's W_img); K, N multiples of 8.  Identical Y and acc.
 * ws: NULL, or a device workspace of at least dqt_fwd_img_workspace_size(T, K,
 * N) bytes (16-byte aligned; DQT_ERR_ARG if smaller).  With it, when the
 * output's 256 x 256 tiles leave the last wave of the 2-SM kernel short, the
 * tiles of that wave are cut into reduction slices whose fp32 partials go to
 * the workspace, and the last slice to finish a region adds them in slice
 * order and applies the epilogue; every partial is an exact integer, so Y and
 * acc are those of the uncut kernel bit for bit.  The size is 0 (any ws) when
 * no cut is planned.  A workspace serves one call at a time. */
size_t dqt_fwd_img_workspace_size(int64_t T, int64_t K, int64_t N);
int dqt_bitlinear_fwd_img(const dqt_bf16* Xq_img, const float* s_x, const dqt_bf16* W_img,
                          float s_w, dqt_grid_t grid, int64_t T, int64_t K, int64_t N,
                          dqt_bf16* Y, int32_t* acc_out, void* ws, size_t ws_bytes,
                          void* stream);

/* Two BitLinear weights that read the same input (a LLaMA MLP's gate and up
 * projections), stacked along N in one call: W_img [N, K] holds the first
 * weight's code image in rows [0, N0) and the second's in rows [N0, N), each
 * with its own per-tensor scale (s_w0, s_w1; Eq. 2-3 apply to each weight
 * alone).  Y [T, N] receives both outputs side by side: columns [0, N0) are
 * the first weight's Y and [N0, N) the second's, bit for bit what two
 * dqt_bitlinear_fwd_img calls write.  N0 a multiple of 256 (whole output
 * tiles), 0 < N0 < N; ws and everything else as dqt_bitlinear_fwd_img. */
int dqt_bitlinear_fwd_img_pair(const dqt_bf16* Xq_img, const float* s_x, const dqt_bf16* W_img,
                               int64_t N0, float s_w0, float s_w1, dqt_grid_t grid, int64_t T,
                               int64_t K, int64_t N, dqt_bf16* Y, int32_t* acc_out, void* ws,
                               size_t ws_bytes, void* stream);

/* Backward w.r.t. the input, no straight-through estimator on the weight
 * (the gradient is taken w.r.t. W_tilde itself, Sec. 3.2):
 *   dX[t,k] = bf16( (sum_n dY[t,n] c[n,k]) * (1 / s_w) )   fp32 accumulation
 *   dY bf16 [T, N];  W int8 [N, K] codes;  dX bf16 [T, K] out.
 * ws: device workspace of at least dqt_bwd_dx_workspace_size(T, N, K) bytes
 * (16-byte aligned; it receives the exact bf16 image of the codes, 3 bytes
 * moved per weight, before the GEMM reads it, and the partials of the
 * last-wave slices, see dqt_bitlinear_bwd_dx_img).  K, N multiples of 8. */
size_t dqt_bwd_dx_workspace_size(int64_t T, int64_t N, int64_t K);
int dqt_bitlinear_bwd_dx(const dqt_bf16* dY, const int8_t* W, float s_w, int64_t T, int64_t N,
                         int64_t K, dqt_bf16* dX, void* ws, size_t ws_bytes, void* stream);

/* The same on the weight's bf16 image W_img [N, K] (dqt_codes_to_bf16).
 * ws: NULL, or at least dqt_bwd_dx_img_workspace_size(T, N, K) bytes
 * (16-byte aligned; DQT_ERR_ARG if smaller): with it the last wave's output
 * tiles may be cut into reduction slices as in dqt_bitlinear_fwd_img, their
 * partials added in slice order (a fixed fp32 summation order, so the result
 * is reproducible; it may differ in the last bits from the uncut kernel's). */
size_t dqt_bwd_dx_img_workspace_size(int64_t T, int64_t N, int64_t K);
int dqt_bitlinear_bwd_dx_img(const dqt_bf16* dY, const dqt_bf16* W_img, float s_w, int64_t T,
                             int64_t N, int64_t K, dqt_bf16* dX, void* ws, size_t ws_bytes,
                             void* stream);

/* The same with dY's rows ldy elements apart (ldy >= N, a multiple of 8):
 * dY may be one weight's columns of a stacked output's gradient (see
 * dqt_bitlinear_bwd_dw_update_img_pair), read in place. */
int dqt_bitlinear_bwd_dx_img_ld(const dqt_bf16* dY, int64_t ldy, const dqt_bf16* W_img, float s_w,
                                int64_t T, int64_t N, int64_t K, dqt_bf16* dX, void* ws,
                                size_t ws_bytes, void* stream);

/* Backward w.r.t. the weight fused with the DQT update (Sec. 3.2, Sec. 4.1, Eq. 5):
 *   X_tilde = bf16(Xq / s_x)                       the dequantised activation
 *   g[n,k]  = sum_t dY[t,n] X_tilde[t,k]           fp32 accumulation in tensor memory
 *   m, v    <- AdamW moments (fp32 [N, K], in place)
 *   x       = c decay - (lr s_w) * m / (sqrt(v) k1 + k2)    (= W' * s_w, see dqt_adamw_t)
 *   c       <- Clip[SR(x), qmin, qmax]  (int8 [N, K], in place; round_mode 1: nearest)
 * The fp32 gradient never reaches memory unless dW_out (fp32 [N, K]) is given
 * (or the workspace holds token-sliced partials, see below).
 * With W, m and v all NULL only dW_out is written (gradient only).
 *   dY bf16 [T, N];  Xq int8 [T, K] and s_x fp32 [T] from dqt_act_quant;
 *   hp, sr: HOST structs.
 *   changed_out: device int64, or NULL; if given, the number of codes that changed
 *   is ADDED to it (the weight-update frequency of Sec. 5.2).
 *   ws: device workspace, 16-byte aligned, of at least the bf16 image of X_tilde
 *   (T K 2 bytes rounded up to 256); dqt_bwd_dw_workspace_size(T, N, K) bytes
 *   also let the GEMM cut token reductions into slices (as for the _img call).
 * K a multiple of 16, N of 8. */
int dqt_bitlinear_bwd_dw_update(const dqt_bf16* dY, const int8_t* Xq, const float* s_x,
                                int8_t* W, float s_w, float* m, float* v, const dqt_adamw_t* hp,
                                const dqt_sr_t* sr, dqt_grid_t grid, int64_t T, int64_t N,
                                int64_t K, float* dW_out, unsigned long long* changed_out,
                                void* ws, size_t ws_bytes, void* stream);
size_t dqt_bwd_dw_workspace_size(int64_t T, int64_t N, int64_t K);

/* The same weight gradient + update on the X_tilde image Xdq bf16 [T, K]
 * (dqt_act_quant_images); ws: the token-slice workspace below, or NULL.
 * W_img_next: NULL, or bf16 [N, K] (16-byte aligned) that receives the exact
 * bf16 image of the updated codes (the next forward's and dX's operand, as
 * dqt_codes_to_bf16 would write it), written by the update itself; it must
 * not be the image any kernel still in flight reads (this step's dX): keep
 * two images and alternate them step by step.  W8_next: NULL, or uint8
 * (16-byte aligned) that receives the E4M3 image of the updated codes (the
 * next FP8 forward's operand), under the same rule: for grids whose codes
 * stay within 16 in magnitude [N, K] as dqt_codes_to_fp8 would write it, for
 * wider grids (6- to 8-bit) the split image [N, 2K] as dqt_codes_to_fp8_split
 * would write it (K a multiple of 16, else DQT_ERR_ALIGN).  Each of the two
 * images needs W, m, v. */
int dqt_bitlinear_bwd_dw_update_img(const dqt_bf16* dY, const dqt_bf16* Xdq, int8_t* W,
                                    float s_w, float* m, float* v, const dqt_adamw_t* hp,
                                    const dqt_sr_t* sr, dqt_grid_t grid, int64_t T, int64_t N,
                                    int64_t K, float* dW_out, dqt_bf16* W_img_next,
                                    uint8_t* W8_next, unsigned long long* changed_out, void* ws,
                                    size_t ws_bytes, void* stream);

/* Workspace (bytes, 16-byte aligned device memory) that lets
 * dqt_bitlinear_bwd_dw_update_img (and the rest of dqt_bitlinear_bwd_dw_update's
 * workspace) cut token reductions into slices:
 *  - a weight gradient whose output is too small to occupy the GPU (few
 *    256 x 256 tiles, long token reduction) is reduced in token slices
 *    throughout;
 *  - otherwise, when the output's tiles do not fill the last wave of SM pairs,
 *    the tiles of that wave are reduced in token slices, so that the last
 *    wave is short.
 * Each slice's fp32 partial goes to the workspace and one streaming pass sums
 * the slices in slice order and applies the update (bit-identical to
 * dqt_sr_update on that summed gradient).  0 = neither applies to this shape
 * on the current device (or under dqt_set_gemm_tiles(1)).  Passing ws = NULL,
 * or fewer bytes, always runs the single fused kernel.  Slicing gives the same
 * update up to the fp32 summation order of the gradient; it is deterministic
 * for a given shape and device. */
size_t dqt_bwd_dw_img_workspace_size(int64_t T, int64_t N, int64_t K);

/* The fused weight gradient and update of two stacked weights that read the
 * same input (see dqt_bitlinear_fwd_img_pair): dY [T, N] holds both outputs'
 * gradients side by side (columns [0, N0) the first weight's), W, m, v [N, K]
 * both weights' codes and moments (rows [0, N0) the first's).  Each weight is
 * updated with its own scale and stochastic-rounding stream: the first with
 * (s_w0, sr0), the second with (s_w1, sr1), its Philox elements counted from
 * its own first element, so codes, m and v equal those of two
 * dqt_bitlinear_bwd_dw_update_img calls computing the same gradients.  N0 a
 * multiple of 256, 0 < N0 < N; ws of dqt_bwd_dw_img_workspace_size(T, N, K)
 * bytes or NULL; W_img_next and W8_next as for dqt_bitlinear_bwd_dw_update_img
 * (both weights' rows); changed_out counts both weights' changed codes. */
int dqt_bitlinear_bwd_dw_update_img_pair(const dqt_bf16* dY, const dqt_bf16* Xdq, int8_t* W,
                                         int64_t N0, float s_w0, float s_w1, float* m, float* v,
                                         const dqt_adamw_t* hp, const dqt_sr_t* sr0,
                                         const dqt_sr_t* sr1, dqt_grid_t grid, int64_t T,
                                         int64_t N, int64_t K, float* dW_out,
                                         dqt_bf16* W_img_next, uint8_t* W8_next,
                                         unsigned long long* changed_out, void* ws,
                                         size_t ws_bytes, void* stream);

/* One weight-gradient + update problem of a grouped call: dY bf16 [T, N],
 * Xdq bf16 [T, K]; W int8, m, v fp32 [N, K] updated in place; N0 = 0 for one
 * weight (s_w0, sr0), or the split of two stacked weights as for
 * dqt_bitlinear_bwd_dw_update_img_pair (rows [0, N0) with s_w0 and sr0, the
 * rest with s_w1 and sr1); W_img_next, W8_next and changed_out as for
 * dqt_bitlinear_bwd_dw_update_img (NULL for none). */
typedef struct {
  const dqt_bf16* dY;
  const dqt_bf16* Xdq;
  int8_t* W;
  float* m;
  float* v;
  int64_t N, K, N0;
  float s_w0, s_w1;
  const dqt_sr_t* sr0;
  const dqt_sr_t* sr1;
  dqt_bf16* W_img_next;
  uint8_t* W8_next;
  unsigned long long* changed_out;
} dqt_dw_problem_t;

/* Two weight-gradient + update problems over the same T tokens (a LLaMA
 * MLP's stacked gate and up, and its down projection) in one persistent
 * launch (Eq. 5 per weight, as dqt_bitlinear_bwd_dw_update_img): the 2-SM
 * CTA pairs walk both problems' 256 x 256 tiles, so together they fill the
 * waves (no token slices, no streaming tail).  Codes, moments, images and
 * counts equal those of the two calls made with ws = NULL, bit for bit.
 * nprob must be 2; hp and grid are the problems' common AdamW constants and
 * grid.  Checks and status codes as for the single calls. */
int dqt_bitlinear_bwd_dw_update_group(const dqt_dw_problem_t* probs, int nprob,
                                      const dqt_adamw_t* hp, dqt_grid_t grid, int64_t T,
                                      void* stream);

/* The AdamW + SR update of dqt_bitlinear_bwd_dw_update for a gradient already
 * in memory (Eq. 5 as a bandwidth-bound stream; 22 bytes per weight):
 *   grad fp32 [numel];  W int8 [numel] in place;  m, v fp32 [numel] in place.
 * Element i uses the uniform of flat index i, so for an [N, K] weight this
 * gives exactly the codes of the fused path for the same fp32 gradient.
 * changed_out as above. */
int dqt_sr_update(const float* grad, int8_t* W, float s_w, float* m, float* v,
                  const dqt_adamw_t* hp, const dqt_sr_t* sr, dqt_grid_t grid, int64_t numel,
                  unsigned long long* changed_out, void* stream);

/* ---- update constants in device memory (CUDA-graph replay) ----------------
 * The AdamW + SR update depends on the step (bias corrections, Philox counter).
 * To replay a captured training step with a new step each time, the update
 * can read its constants from device memory when the kernel runs:
 *   dqt_update_consts derives, on the host, the block the update kernels use
 *   (the constants listed at dqt_adamw_t, the grid, s_w and the SR key) into
 *   `out` (host memory, at least dqt_update_consts_size() bytes); the caller
 *   copies it to a 16-byte aligned device buffer ordered before the launch
 *   (e.g. a cudaMemcpyAsync from pinned memory captured in the same graph).
 * The _dev entry points are dqt_bitlinear_bwd_dw_update_img and dqt_sr_update
 * with (hp, sr, grid, s_w) replaced by that device block; results are
 * identical for identical constants.  W, m, v are required; the weight
 * gradient takes the X_tilde image Xdq, the token-slice workspace and the
 * next-step images W_img_next / W8_next of dqt_bitlinear_bwd_dw_update_img
 * (W8_next the direct image [N, K] only, for grids within 16 in magnitude:
 * the grid is in the device block, so this call can neither check it nor
 * choose the split image). */
size_t dqt_update_consts_size(void);
int dqt_update_consts(const dqt_adamw_t* hp, const dqt_sr_t* sr, dqt_grid_t grid, float s_w,
                      void* out, size_t out_bytes);
int dqt_bitlinear_bwd_dw_update_dev(const dqt_bf16* dY, const dqt_bf16* Xdq, int8_t* W, float* m,
                                    float* v, const void* consts_dev, int64_t T, int64_t N,
                                    int64_t K, float* dW_out, dqt_bf16* W_img_next,
                                    uint8_t* W8_next, unsigned long long* changed_out, void* ws,
                                    size_t ws_bytes, void* stream);
int dqt_sr_update_dev(const float* grad, int8_t* W, float* m, float* v, const void* consts_dev,
                      int64_t numel, unsigned long long* changed_out, void* stream);

/* ---- FP8 environment (Sec. 4.1 hardware paragraph; Sec. 4.3) ------------------
 * The paper also trains DQT models with 8-bit floating-point GEMM operands.
 * These three calls are the forward of that variant; the backward uses the
 * bf16 calls above (dX with dqt_codes_to_bf16's image, dW + update with the
 * Xdq image written here).  An E4M3 byte is the OCP 8-bit float "e4m3fn":
 * sign, 4 exponent bits (bias 7), 3 mantissa bits, largest finite 448.
 *
 * Activations, per token t:
 *   amax[t] = max_k |X[t,k]|,  s_x8[t] = 448 / max(amax[t], 1e-5)   (fp32 divide)
 *   Xq8[t,k] = E4M3(X[t,k] * s_x8[t])   fp32 multiply, round-to-nearest-even,
 *                                       saturating at +-448, sign kept for zero
 *   X    bf16 [T, K] in;  Xq8 uint8 [T, K] out (required);  s_x8 fp32 [T] out
 *   Xdq  bf16 [T, K] out, or NULL: bf16(value(Xq8) / s_x8), the dequantised
 *        activation the weight gradient uses
 * K a multiple of 16 (16-byte E4M3 rows). */
int dqt_act_quant_fp8(const dqt_bf16* X, int64_t T, int64_t K, uint8_t* Xq8, float* s_x8,
                      dqt_bf16* Xdq, void* stream);

/* E4M3 image of weight codes: W8[i] = E4M3(W[i]), exact because every integer
 * of magnitude <= 16 is an E4M3 value.  The grid bounds the codes: grids
 * with a code beyond 16 in magnitude (6- to 8-bit) return DQT_ERR_RANGE (their
 * E4M3 form is dqt_codes_to_fp8_split).  numel >= 1. */
int dqt_codes_to_fp8(const int8_t* W, int64_t numel, dqt_grid_t grid, uint8_t* W8, void* stream);

/* E4M3 split image of codes of any width, for the FP8 forward of 6- to 8-bit
 * grids: each code c = 16 h + l with h = c >> 4 (floor(c / 16), in [-8, 7])
 * and l = c & 15 (in [0, 15]); 16 h and l are E4M3 values, so both halves
 * are exact.  W int8 [N, K] -> W8 uint8 [N, 2K]: row n holds E4M3(16 h) of
 * its K codes, then E4M3(l).  K a multiple of 16. */
int dqt_codes_to_fp8_split(const int8_t* W, int64_t N, int64_t K, uint8_t* W8, void* stream);

/* Forward on E4M3 operands (tcgen05 kind::f8f6f4, fp32 accumulation):
 *   acc[t,n] = sum_k value(Xq8[t,k]) * c[n,k]       fp32 accumulator
 *   Y[t,n]   = bf16( acc * (1 / (s_x8[t] * s_w)) )
 * Each product is exact; the sum is rounded by the fp32 accumulation (in an
 * order the hardware chooses), so Y equals the exact-sum formula up to that
 * rounding.  Xq8 uint8 [T, K], s_x8 fp32 [T] (dqt_act_quant_fp8); W8 uint8
 * [N, K] (dqt_codes_to_fp8) for grids within 16 in magnitude; Y bf16 [T, N]
 * out; acc_out fp32 [T, N] out, or NULL.  K a multiple of 16, N of 8.
 * Grids beyond 16 (6- to 8-bit): W8 is the split image uint8 [N, 2K]
 * (dqt_codes_to_fp8_split) and the sum runs over both halves, the activation
 * row read for each: acc = sum_k value(Xq8[t,k]) 16 h[n,k] + value(Xq8[t,k])
 * l[n,k], 2K exact products accumulated in fp32; K a multiple of 128. */
int dqt_bitlinear_fwd_fp8(const uint8_t* Xq8, const float* s_x8, const uint8_t* W8, float s_w,
                          dqt_grid_t grid, int64_t T, int64_t K, int64_t N, dqt_bf16* Y,
                          float* acc_out, void* stream);

/* dqt_bitlinear_fwd_fp8 for two stacked weights that read the same input (a
 * LLaMA MLP's gate and up projections): W8 uint8 [N, K] holds both weights'
 * E4M3 images (rows [0, N0) the first's), Y bf16 [T, N] both outputs side by
 * side, the columns [0, N0) scaled with s_w0 and the rest with s_w1: Y and
 * acc_out equal two dqt_bitlinear_fwd_fp8 calls', bit for bit.  N0 a multiple
 * of 256, 0 < N0 < N; the rest (the split image of wide grids included) as
 * for dqt_bitlinear_fwd_fp8. */
int dqt_bitlinear_fwd_fp8_pair(const uint8_t* Xq8, const float* s_x8, const uint8_t* W8, int64_t N0,
                               float s_w0, float s_w1, dqt_grid_t grid, int64_t T, int64_t K,
                               int64_t N, dqt_bf16* Y, float* acc_out, void* stream);

/* ---- 2-bit packed ternary codes (Sec. 1: ternary weights need a fraction of
 * a byte each; 4 codes per byte here, 0.25 GB per 1B weights) ----------------
 * Code e of a tensor is field e % 4 (bits 2 (e % 4) and 2 (e % 4) + 1) of byte
 * e / 4, a 2-bit two's-complement number (-1 = 0b11, 0 = 0b00, +1 = 0b01);
 * unused fields of the last byte are 0.  A packed [N, K] weight needs K % 4 ==
 * 0 (K % 8 == 0 for the GEMMs) so that rows start on byte boundaries.  Packed
 * tensors are ceil(numel / 4) bytes, 16-byte aligned. */
int dqt_pack_ternary(const int8_t* codes, int64_t numel, uint8_t* packed, void* stream);
int dqt_unpack_ternary(const uint8_t* packed, int64_t numel, int8_t* codes, void* stream);
/* GEMM operand images straight from packed codes (as dqt_codes_to_bf16 and
 * dqt_codes_to_fp8 do from int8 codes). */
int dqt_packed_to_bf16(const uint8_t* packed, int64_t numel, dqt_bf16* W_img, void* stream);
int dqt_packed_to_fp8(const uint8_t* packed, int64_t numel, uint8_t* W8, void* stream);
/* dqt_sr_update and dqt_bitlinear_bwd_dw_update_img (X_tilde image Xdq,
 * token-slice workspace) on packed ternary codes (the grid is [-1, 1]);
 * identical results, 0.25 byte per weight of code traffic. */
int dqt_sr_update_packed(const float* grad, uint8_t* Wp, float s_w, float* m, float* v,
                         const dqt_adamw_t* hp, const dqt_sr_t* sr, int64_t numel,
                         unsigned long long* changed_out, void* stream);
int dqt_bitlinear_bwd_dw_update_packed(const dqt_bf16* dY, const dqt_bf16* Xdq, uint8_t* Wp,
                                       float s_w, float* m, float* v, const dqt_adamw_t* hp,
                                       const dqt_sr_t* sr, int64_t T, int64_t N, int64_t K,
                                       float* dW_out, unsigned long long* changed_out, void* ws,
                                       size_t ws_bytes, void* stream);

/* ---- Adafactor with stochastic rounding (Sec. 4.3) ---------------------------
 * The memory-efficient optimiser the paper pairs with DQT: Adafactor (Shazeer
 * & Stern, ICML 2018) without first moment keeps only the row means R [N] and
 * column means C [K] of an N x K weight's squared gradient (fp32, zero at the
 * start, in place), so no per-weight optimiser state exists at all.  Step t:
 *   b2 = 1 - t^decay_rate;  rho = relative_step ? min(warmup_init ? 1e-6 t : 1e-2,
 *                                                  1/sqrt(t)) : lr
 *   R <- b2 R + (1 - b2) mean_k(g^2 + eps1);  C <- b2 C + (1 - b2) mean_n(g^2 + eps1)
 *   Rbar = mean R; the inverse square root of the rank-one estimate R C / Rbar is
 *   a row factor a[n] = 1 / sqrt(R[n] / Rbar) times a column factor
 *   b[k] = 1 / sqrt(C[k]) (each two correctly rounded fp32 operations);
 *   u = (g a[n]) b[k]
 *   alpha = rho * (scale_parameter ? max(eps2, RMS(W)) : 1),  RMS(W) = RMS(c) / s_w
 *   x = c (1 - weight_decay alpha) - s_w alpha / max(1, RMS(u) / clip_d) * u
 *   c <- Clip[SR(x), qmin, qmax]   (Eq. 1, Eq. 5; the Philox stream of dqt_sr_t
 *                                   with counter step t, as for AdamW)
 * Defaults a caller may start from: lr 1e-3, eps1 1e-30, eps2 1e-3, clip_d 1,
 * decay_rate -0.8, weight_decay 0, relative_step 0, scale_parameter 0. */
typedef struct {
  float lr, eps1, eps2, clip_d, decay_rate, weight_decay;
  int64_t step; /* t >= 1 */
  int32_t relative_step, scale_parameter, warmup_init, pad;
} dqt_adafactor_t;

/* Statistics of one step for a gradient G fp32 [N, K] in memory: updates R, C,
 * writes the factors a_out fp32 [N] and b_out fp32 [K], and 8 floats to
 * scalars_out (device, 16-byte aligned): {Rbar, code-domain step
 * s_w alpha / max(1, RMS(u)/clip_d), decay 1 - weight_decay alpha, RMS(u),
 * RMS(W) (0 unless scale_parameter: the codes are not read then), alpha, 0, 0}.
 * W: the codes before the step (int8 [N, K], or packed ternary if `packed`).  Workspace: dqt_adafactor_workspace_size(N, K) bytes,
 * 256-byte aligned.  Every sum has a fixed order: deterministic. */
size_t dqt_adafactor_workspace_size(int64_t N, int64_t K);
int dqt_adafactor_stats(const float* G, const void* W, int32_t packed, float s_w, float* R,
                        float* C, const dqt_adafactor_t* hp, int64_t N, int64_t K, float* a_out,
                        float* b_out, float* scalars_out, void* ws, size_t ws_bytes,
                        void* stream);
/* The per-element step given the factors a [N], b [K] and the scalars
 * {., step, decay} in device memory (as dqt_adafactor_stats writes them):
 * u = (g a[n]) b[k], x = c decay - step u, each a separately rounded fp32
 * operation, then SR with counter `step_t` and the clamp.  changed_out as for
 * dqt_sr_update. */
int dqt_adafactor_apply(const float* G, void* W, int32_t packed, const float* a, const float* b,
                        const float* scalars, int64_t step_t, const dqt_sr_t* sr, dqt_grid_t grid,
                        int64_t N, int64_t K, unsigned long long* changed_out, void* stream);
/* The whole backward-and-update of a BitLinear weight with Adafactor: the
 * weight gradient dY^T Xdq (fp32, tensor cores; Xdq the X_tilde image of
 * dqt_act_quant_images) into the workspace, then the
 * statistics and the per-element step above.  Workspace:
 * dqt_bwd_dw_adafactor_workspace_size(T, N, K) bytes (the fp32 gradient, the
 * statistics, and token-slice partials when the GEMM splits the reduction). */
size_t dqt_bwd_dw_adafactor_workspace_size(int64_t T, int64_t N, int64_t K);
int dqt_bitlinear_bwd_dw_adafactor(const dqt_bf16* dY, const dqt_bf16* Xdq, void* W,
                                   int32_t packed, float s_w, float* R, float* C,
                                   const dqt_adafactor_t* hp, const dqt_sr_t* sr, dqt_grid_t grid,
                                   int64_t T, int64_t N, int64_t K,
                                   unsigned long long* changed_out, void* ws, size_t ws_bytes,
                                   void* stream);

/* ---------------------------------------------------------------------------
 * Decoder support.  Not part of the DQT method: two operations of the
 * LLaMA-structured decoder built around the BitLinear layers (the model family
 * of Sec. 4.1), each one pass over bf16 data in HBM with fp32 arithmetic.
 * ------------------------------------------------------------------------- */

/* Rotary position embedding (LLaMA form) of x, bf16 [rows, H, D] contiguous
 * with rows = B * S (row r is at position r % S), into y (same shape; y must
 * not overlap x).  Each interleaved pair (x[2i], x[2i+1]) of a head is a
 * complex number multiplied by exp(i theta_{pos, i}):
 *   y[2i] = x[2i] c - x[2i+1] s,   y[2i+1] = x[2i] s + x[2i+1] c
 * with (c, s) = cos_sin[pos, i, 0..1], fp32 [S, D/2, 2] supplied by the
 * caller; each product and sum is a separately rounded fp32 operation, the
 * result rounded to bf16 (nearest-even).  inverse = 1 rotates by -theta (the
 * backward: the transpose of the rotation).  D a multiple of 8; x, y, cos_sin
 * 16-byte aligned (DQT_ERR_ALIGN otherwise). */
int dqt_rope_bf16(const dqt_bf16* x, dqt_bf16* y, const float* cos_sin, int64_t rows, int64_t S,
                  int64_t H, int64_t D, int32_t inverse, void* stream);

/* Token cross-entropy over bf16 logits [M, V] (row-major, V a multiple of 8,
 * 16-byte aligned) with int64 targets [M]: per row, in fp32,
 *   lse[m] = log sum_v exp(logits[m, v]),   row_loss[m] = lse[m] - logits[m, t_m]
 * (row_loss 0 for a target outside [0, V)).  The mean loss is the caller's sum
 * of row_loss over the rows with valid targets divided by their count. */
int dqt_cross_entropy_fwd_bf16(const dqt_bf16* logits, const int64_t* targets, int64_t M,
                               int64_t V, float* lse, float* row_loss, void* stream);
/* Its gradient: dlogits[m, v] = bf16((exp(logits[m, v] - lse[m]) - [v == t_m]) * scale[0]),
 * scale a device fp32 scalar (the upstream gradient divided by the count of
 * valid rows); rows with a target outside [0, V) get zeros.  dlogits 16-byte
 * aligned, [M, V] bf16, not overlapping logits. */
int dqt_cross_entropy_bwd_bf16(const dqt_bf16* logits, const int64_t* targets, const float* lse,
                               const float* scale, int64_t M, int64_t V, dqt_bf16* dlogits,
                               void* stream);

/* SwiGLU gate of the decoder's MLP: h = silu(g) u = g sigmoid(g) u per
 * element of bf16 g, u [n], evaluated in fp32 and rounded once to bf16.  Its
 * backward, with s = sigmoid(g):  dg = dh u s (1 + g (1 - s)),  du = dh g s
 * (fp32, each rounded once to bf16).  n a multiple of 8, every pointer 16-byte
 * aligned, outputs not overlapping inputs. */
int dqt_swiglu_bf16(const dqt_bf16* g, const dqt_bf16* u, dqt_bf16* h, int64_t n, void* stream);
int dqt_swiglu_bwd_bf16(const dqt_bf16* g, const dqt_bf16* u, const dqt_bf16* dh, dqt_bf16* dg,
                        dqt_bf16* du, int64_t n, void* stream);

/* RMSNorm of the decoder: per row of x bf16 [rows, D],
 *   rstd = 1 / sqrt(mean_j x_j^2 + eps),   y_j = x_j rstd w_j
 * in fp32, y rounded once to bf16; rstd fp32 [rows] is kept for the backward.
 * D a multiple of 8 and at most 2048 (DQT_ERR_RANGE beyond); x, w, y 16-byte
 * aligned. */
int dqt_rmsnorm_bf16(const dqt_bf16* x, const dqt_bf16* w, float eps, int64_t rows, int64_t D,
                     dqt_bf16* y, float* rstd, void* stream);
/* Its backward for the upstream gradient dy [rows, D]:
 *   dx_j = rstd w_j dy_j - x_j rstd^3 (1/D) sum_k w_k dy_k x_k   (bf16 [rows, D])
 *   dw_j = sum over rows of dy_j x_j rstd                        (bf16 [D])
 * dw is summed in a fixed order (per-warp partial sums in the workspace, then
 * a column reduction), so it is deterministic.  Workspace:
 * dqt_rmsnorm_bwd_workspace_size(rows, D) bytes for the current device,
 * 16-byte aligned. */
size_t dqt_rmsnorm_bwd_workspace_size(int64_t rows, int64_t D);
int dqt_rmsnorm_bwd_bf16(const dqt_bf16* x, const dqt_bf16* w, const float* rstd,
                         const dqt_bf16* dy, int64_t rows, int64_t D, dqt_bf16* dx, dqt_bf16* dw,
                         void* ws, size_t ws_bytes, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* DQT_H_ */

// Host-side interfaces between the C ABI (dqt_api.cu) and the kernel files.
#pragma once

#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "../../include/dqt.h"
#include "dqt_device.cuh"

namespace dqt {

// Argument rules shared by entry points that must accept and reject alike.
// A weight grid: Q_n <= 0 <= Q_p, both within int8.
inline bool grid_ok(dqt_grid_t g) {
  return g.qmin <= g.qmax && g.qmin >= -128 && g.qmax <= 127 && g.qmin <= 0 && g.qmax >= 0;
}
// The AbsMean of Eq. 2 must be positive and finite for s_w = Q_p / AbsMean.
inline bool absmean_ok(double absmean) { return absmean > 0.0 && isfinite(absmean); }

// Largest wait, in ns, a kernel makes before it records a timeout.
uint64_t wait_limit_ns();

// Device address of the current device's status word (NULL on failure).
unsigned int* status_word();

// GEMM kernel selection: 0 = 2-SM pair tiles where possible, 1 = 1-SM tiles.
int gemm_mode();

enum GemmKind { GEMM_FWD = 0, GEMM_DX = 1, GEMM_DW = 2, GEMM_FWD8 = 3 };

struct GemmLaunch {
  GemmKind kind;
  // Output is M x N, reduced over Kred.
  int M, N, Kred;
  // Operands (bf16, row-major, contiguous):
  //   FWD: A = Xq_img [M=T, Kred=K],  B = W_img [N, Kred=K]     (both K-major)
  //   DX : A = dY     [M=T, Kred=N],  B = W_img [Kred=N, N=K]   (B MN-major)
  //   DW : A = dY     [Kred=T, M=N],  B = Xdq   [Kred=T, N=K]   (both MN-major)
  //   FWD8: A = Xq8 [M=T, Kred=K], B = W8 [N, Kred=K], E4M3 bytes (both K-major)
  const void* A;
  const void* B;
  int chunk_k;  // FWD: reduction elements per exact fp32 chunk (multiple of 64)
  bool pair;    // use the 2-SM (cta_group::2) kernel (not with drained chunks)
  // Epilogue operands.
  const float* s_x;  // FWD, FWD8
  float scale;       // FWD: s_w; DX: 1/s_w
  void* out_bf16;    // FWD: Y; DX: dX
  int32_t* acc_out;  // FWD, optional
  float* acc_f32;    // FWD8, optional
  int8_t* W;         // DW (with m, v), optional; 2-bit packed ternary bytes if `packed`
  bool packed;
  float* m;
  float* v;
  float* dW_out;  // DW, optional
  unsigned long long* changed;
  UpdateConsts uc;
  const UpdateConsts* uc_dev;  // DW: read the update constants from device memory if set
  void* ws;                    // DW: split-T workspace (fp32 slabs), or NULL
  size_t ws_bytes;
  // two stacked weights (2-SM kernels only): from output column (FWD) or
  // output row (DW) `split` on (a multiple of 256) the second weight, with
  // scale scale1 (FWD) or constants uc1 (DW); 0: one weight
  int split;
  float scale1;
  UpdateConsts uc1;
  int64_t lda;  // DX: elements between rows of A (dY); 0: packed rows
  void* img_next;   // DW: bf16 image of the updated codes, or NULL
  void* img8_next;  // DW: E4M3 image of the updated codes, or NULL
  // DW: img8_next is the split image [M, 2 N] (16 (c >> 4), then c & 15 in
  // each row) of codes wider than E4M3's exact integers
  bool img8_split;
  // FWD8 on split codes: B is [N, Kred = 2 a_wrap] (each code c as 16 (c >> 4)
  // in the first half of its row and c & 15 in the second) and A [M, a_wrap]
  // is read twice, k-block kb from column (kb * 128) mod a_wrap; 0: no split
  int a_wrap;
};

// Token slices the 2-SM dW GEMM of an M x N output reduced over Kred uses
// when given a workspace of dw_splits * M * N floats (1 = no split).
int dw_splits(int M, int N, int Kred);

// The last-wave tail of a 2-SM dW GEMM on `clusters` clusters: `tail` tiles
// (tile indices full .. full + tail - 1) each cut into `splits` token slices
// of `kbps` k-blocks; `bytes` of workspace for their partials (splits 0: no
// tail split).
struct TailPlan {
  int splits, tail, full, kbps;
  size_t bytes;
};
TailPlan tail_plan(int M, int N, int Kred, int clusters);

// Workspace bytes for the last-wave token (or reduction) slices of a 2-SM
// GEMM with an M x N output reduced over Kred on this device: the slices'
// fp32 partials, or 0 when the output's tiles fill the waves closely enough
// that no slicing is planned.
size_t gemm_tail_bytes(int M, int N, int Kred);

// Sums the tail slices' partials (slice s of tail tile j at (s * tail + j) *
// 65536 floats, tile-local row-major 256 x 256; tile full + j of an M x N
// output with num_n tiles per row) in slice order and applies the update of
// sr_update_kernel to W, m, v (if W) at the global element indices, and/or
// writes the summed gradient to dW_out.  img8_split: img8_next is the split
// E4M3 image, rows of 2 N bytes.
int launch_tail_update(const float* part, int splits, int tail, int full, int num_n, int M, int N,
                       int8_t* W, bool packed, float* m, float* v, const UpdateConsts& uc,
                       const UpdateConsts* uc_dev, unsigned long long* changed, float* dW_out,
                       cudaStream_t stream, const UpdateConsts* uc1 = nullptr, int split = 0,
                       bool col_major = false, uint16_t* img_next = nullptr,
                       uint8_t* img8_next = nullptr, bool img8_split = false);

// Sum `splits` fp32 slabs (stride `slab` elements) in slice order and apply
// the update to W, m, v (numel elements); optionally write the sum to g_out
// and the bf16 / E4M3 images of the new codes to img / img8 (int8 codes);
// img8_k > 0: img8 is the split E4M3 image of rows of img8_k codes (2 img8_k
// bytes each: 16 (c >> 4), then c & 15), numel a multiple of img8_k.
int launch_sr_update_slabs(const float* slabs, int splits, long long slab, int8_t* W, float* m,
                           float* v, int64_t numel, const UpdateConsts& uc,
                           const UpdateConsts* uc_dev, unsigned long long* changed, float* g_out,
                           cudaStream_t stream, bool packed = false, uint16_t* img = nullptr,
                           uint8_t* img8 = nullptr, int64_t img8_k = 0);
// Sum the slabs into out (gradient only).
int launch_slab_sum(const float* slabs, int splits, long long slab, float* out,
                    cudaStream_t stream);

int launch_gemm(const GemmLaunch& g, cudaStream_t stream);
// Two 2-SM dW + update launches (kind GEMM_DW, int8 codes with W, m, v,
// constants by value, the same reduction length Kred) as one persistent
// launch over both problems' whole tiles; dW_out, stacked weights (split)
// and the next-step images as for launch_gemm.  Nonzero on an unsupported
// launch record (1) or a CUDA error (3).
int launch_dw_group(const GemmLaunch& g0, const GemmLaunch& g1, cudaStream_t stream);

int launch_act_quant(const uint16_t* X, int64_t T, int64_t K, int8_t* Xq, float* s_x,
                     uint16_t* Xq_img, uint16_t* Xdq, cudaStream_t stream);
int launch_codes_to_bf16(const int8_t* W, int64_t numel, uint16_t* W_img, cudaStream_t stream);
// Xdq[t,k] = bf16(Xq[t,k] / s_x[t]) (the image dqt_act_quant writes); K % 16 == 0.
int launch_codes_to_xdq(const int8_t* Xq, const float* s_x, int64_t T, int64_t K, uint16_t* Xdq,
                        cudaStream_t stream);
// FP8 environment: E4M3 activations with per-token scale 448 / max(amax, 1e-5)
// (and optionally the dequantised bf16 image), and E4M3 images of weight codes.
int launch_act_quant_fp8(const uint16_t* X, int64_t T, int64_t K, uint8_t* Xq8, float* s8,
                         uint16_t* Xdq, cudaStream_t stream);
int launch_codes_to_fp8(const int8_t* W, int64_t numel, uint8_t* W8, cudaStream_t stream);
// E4M3 split image of codes [N, K] (K % 16 == 0): W8 [N, 2K], row n holds
// 16 (c >> 4) for every code of row n, then c & 15 (both exact in E4M3).
int launch_codes_to_fp8_split(const int8_t* W, int64_t N, int64_t K, uint8_t* W8,
                              cudaStream_t stream);
int launch_absmean_partial(const float* W0, int64_t numel, double* ws, cudaStream_t stream);
int launch_absmean_codes(const float* W0, int64_t numel, float s_w, int32_t qmin, int32_t qmax,
                         int8_t* codes, cudaStream_t stream);
constexpr int kAbsmeanBlocks = 1024;

// Decoder support (rotary embedding, token cross-entropy): decoder_ops.cu.
int launch_rope(const uint16_t* x, uint16_t* y, const float* cos_sin, int64_t rows, int64_t S,
                int64_t H, int64_t D, bool inverse, cudaStream_t stream);
int launch_ce_fwd(const uint16_t* logits, const int64_t* targets, int64_t M, int64_t V,
                  float* lse, float* row_loss, cudaStream_t stream);
int launch_ce_bwd(const uint16_t* logits, const int64_t* targets, const float* lse,
                  const float* scale, int64_t M, int64_t V, uint16_t* dlogits,
                  cudaStream_t stream);
int launch_swiglu(const uint16_t* g, const uint16_t* u, uint16_t* h, int64_t n,
                  cudaStream_t stream);
int launch_swiglu_bwd(const uint16_t* g, const uint16_t* u, const uint16_t* dh, uint16_t* dg,
                      uint16_t* du, int64_t n, cudaStream_t stream);
int launch_rmsnorm(const uint16_t* x, const uint16_t* w, float eps, int64_t rows, int64_t D,
                   uint16_t* y, float* rstd, cudaStream_t stream);
size_t rmsnorm_bwd_ws(int64_t rows, int64_t D);
int launch_rmsnorm_bwd(const uint16_t* x, const uint16_t* w, const float* rstd,
                       const uint16_t* dy, int64_t rows, int64_t D, uint16_t* dx, uint16_t* dw,
                       float* part, cudaStream_t stream);

// 2-bit packed ternary codes (4 per byte): conversions and operand images.
int launch_pack_ternary(const int8_t* c, int64_t n, uint8_t* out, cudaStream_t stream);
int launch_unpack_ternary(const uint8_t* p, int64_t n, int8_t* c, cudaStream_t stream);
int launch_packed_to_bf16(const uint8_t* p, int64_t n, uint16_t* img, cudaStream_t stream);
int launch_packed_to_fp8(const uint8_t* p, int64_t n, uint8_t* out, cudaStream_t stream);

// Adafactor (factored second moment, no first moment) host-derived constants.
struct AdafactorConsts {
  float b2, omb2, rho, eps1, eps2, clip_d, weight_decay;
  int32_t scale_parameter;
};
// Workspace of the statistics passes for an N x K weight; it also holds a
// set of factor vectors and a scalar block (adafactor_bufs) for callers that
// do not keep their own.
size_t adafactor_stats_ws(int64_t N, int64_t K);
struct AdafactorBufs {
  float* a;        // [N] row factors
  float* b;        // [K] column factors
  float* scalars;  // [8]
};
AdafactorBufs adafactor_bufs(void* ws, int64_t N, int64_t K);
// R, C updated in place; a_out [N], b_out [K] get the inverse-square-root
// factors, scalars_out (8 floats) {Rbar, code-domain step, decay, rms_u,
// rms_x, alpha}.
int launch_adafactor_stats(const float* G, const int8_t* W, bool packed, float s_w, float* R,
                           float* C, const AdafactorConsts& h, int64_t N, int64_t K, void* ws,
                           float* a_out, float* b_out, float* scalars_out, cudaStream_t stream);
// The per-element update given the factors and scalars {., step, decay}
// (device).  Uses the grid, round mode and Philox key/counter fields of uc.
int launch_adafactor_apply(const float* G, int8_t* W, bool packed, const float* fa,
                           const float* fb, const float* scalars, const UpdateConsts& uc,
                           int64_t N, int64_t K, unsigned long long* changed,
                           cudaStream_t stream);

int launch_sr_update(const float* grad, int8_t* W, float* m, float* v, int64_t numel,
                     const UpdateConsts& uc, const UpdateConsts* uc_dev,
                     unsigned long long* changed, cudaStream_t stream, bool packed = false);

}  // namespace dqt

// C ABI of the DQT library (declared in include/dqt.h): argument checks,
// host-side derivation of the AdamW constants, and kernel launches.
#include <math.h>
#include <stdint.h>
#include <string.h>

#include <atomic>

#include "../../include/dqt.h"
#include "dqt_internal.h"

namespace dqt {

// One status word per device (bounded-wait timeouts, see dqt_device.cuh).
__device__ unsigned int g_status_word;

namespace {
std::atomic<uint64_t> g_wait_ns{2000000000ull};
std::atomic<int> g_gemm_mode{0};
constexpr int kMaxDevices = 64;
// Per-device address cache; host threads may look it up concurrently.
std::atomic<unsigned int*> g_status_ptr[kMaxDevices] = {};
}  // namespace

uint64_t wait_limit_ns() { return g_wait_ns.load(); }
int gemm_mode() { return g_gemm_mode.load(); }

unsigned int* status_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  unsigned int* cached = g_status_ptr[dev].load(std::memory_order_relaxed);
  if (!cached) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
    cached = static_cast<unsigned int*>(p);
    g_status_ptr[dev].store(cached, std::memory_order_relaxed);
  }
  return cached;
}

}  // namespace dqt

namespace {

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

using dqt::grid_ok;

inline cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

// AdamW and SR constants, derived on the host in fp64 and rounded once to fp32.
int make_update_consts(const dqt_adamw_t* hp, const dqt_sr_t* sr, dqt_grid_t g, float s_w,
                       dqt::UpdateConsts* uc) {
  if (!hp || !sr || !grid_ok(g)) return DQT_ERR_ARG;
  if (hp->step < 1 || !(hp->beta1 >= 0.0f && hp->beta1 < 1.0f) ||
      !(hp->beta2 >= 0.0f && hp->beta2 < 1.0f) || !(hp->eps > 0.0f) || !(hp->lr >= 0.0f) ||
      !isfinite(hp->weight_decay) || !(s_w > 0.0f) || !isfinite(s_w))
    return DQT_ERR_ARG;
  if (sr->round_mode != 0 && sr->round_mode != 1) return DQT_ERR_ARG;
  if (sr->elem0 < 0) return DQT_ERR_ARG;
  if (sr->elem0 & 3) return DQT_ERR_ALIGN;
  const double b1 = hp->beta1, b2 = hp->beta2, st = static_cast<double>(hp->step);
  const double bc1 = 1.0 - pow(b1, st), bc2 = 1.0 - pow(b2, st);
  if (!(bc1 > 0.0) || !(bc2 > 0.0)) return DQT_ERR_ARG;
  uc->b1 = hp->beta1;
  uc->b2 = hp->beta2;
  uc->omb1 = static_cast<float>(1.0 - b1);
  uc->omb2 = static_cast<float>(1.0 - b2);
  uc->k1 = static_cast<float>(bc1 / sqrt(bc2));
  uc->k2 = static_cast<float>(bc1 * static_cast<double>(hp->eps));
  uc->decay = static_cast<float>(1.0 - static_cast<double>(hp->lr) * hp->weight_decay);
  uc->lrs = static_cast<float>(static_cast<double>(hp->lr) * static_cast<double>(s_w));
  if (!(uc->k1 > 0.0f) || !(uc->k2 > 0.0f)) return DQT_ERR_ARG;
  uc->qmin = g.qmin;
  uc->qmax = g.qmax;
  uc->step_lo = static_cast<uint32_t>(hp->step);
  uc->tensor_id = sr->tensor_id;
  uc->key0 = static_cast<uint32_t>(sr->seed);
  uc->key1 = static_cast<uint32_t>(sr->seed >> 32);
  uc->round_mode = sr->round_mode;
  const uint64_t blk0 = static_cast<uint64_t>(sr->elem0) >> 2;
  uc->blk0_lo = static_cast<uint32_t>(blk0);
  uc->blk0_hi = static_cast<uint32_t>(blk0 >> 32);
  return DQT_OK;
}

constexpr int64_t kMaxDim = (int64_t(1) << 31) - 1;

}  // namespace

extern "C" {

const char* dqt_status_string(int s) {
  switch (s) {
    case DQT_OK: return "DQT_OK";
    case DQT_ERR_ARG: return "DQT_ERR_ARG: invalid argument";
    case DQT_ERR_ALIGN: return "DQT_ERR_ALIGN: pointer not 16-byte aligned or K/N not a multiple of 8";
    case DQT_ERR_CUDA: return "DQT_ERR_CUDA: CUDA call failed";
    case DQT_ERR_TIMEOUT: return "DQT_ERR_TIMEOUT: a bounded device wait ran out";
    case DQT_ERR_RANGE: return "DQT_ERR_RANGE: size out of the supported range";
    default: return "DQT: unknown status";
  }
}

int dqt_grid_for_bits(float bits, dqt_grid_t* out) {
  if (!out) return DQT_ERR_ARG;
  if (fabsf(bits - 1.58f) < 1e-3f) {
    out->qmin = -1;
    out->qmax = 1;
    return DQT_OK;
  }
  const float r = rintf(bits);
  if (r != bits || r < 2.0f || r > 8.0f) return DQT_ERR_ARG;
  const int n = static_cast<int>(r);
  out->qmin = -(1 << (n - 1));
  out->qmax = (1 << (n - 1)) - 1;
  return DQT_OK;
}

int dqt_set_wait_limit_ns(uint64_t ns) {
  dqt::g_wait_ns.store(ns);
  return DQT_OK;
}

int dqt_set_gemm_tiles(int mode) {
  if (mode != 0 && mode != 1) return DQT_ERR_ARG;
  dqt::g_gemm_mode.store(mode);
  return DQT_OK;
}

int dqt_check_device_status(void* stream) {
  if (cudaStreamSynchronize(as_stream(stream)) != cudaSuccess) return DQT_ERR_CUDA;
  unsigned int* p = dqt::status_word();
  if (!p) return DQT_ERR_CUDA;
  unsigned int h = 0;
  if (cudaMemcpy(&h, p, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess) return DQT_ERR_CUDA;
  if (h != 0) {
    const unsigned int zero = 0;
    if (cudaMemcpy(p, &zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess)
      return DQT_ERR_CUDA;
    return DQT_ERR_TIMEOUT;
  }
  return DQT_OK;
}

size_t dqt_absmean_workspace_size(void) { return (dqt::kAbsmeanBlocks + 1) * sizeof(double); }

int dqt_absmean_init(const float* W0, int64_t numel, dqt_grid_t grid, int8_t* codes, float* s_w,
                     void* ws, size_t ws_bytes, void* stream) {
  if (!W0 || !codes || !s_w || !ws || numel <= 0 || !grid_ok(grid) || grid.qmax <= 0)
    return DQT_ERR_ARG;
  if (ws_bytes < dqt_absmean_workspace_size()) return DQT_ERR_ARG;
  if ((reinterpret_cast<uintptr_t>(ws) & 7u) != 0) return DQT_ERR_ALIGN;
  cudaStream_t st = as_stream(stream);
  double* dws = static_cast<double*>(ws);
  if (dqt::launch_absmean_partial(W0, numel, dws, st)) return DQT_ERR_CUDA;
  double sum = 0.0;
  if (cudaMemcpyAsync(&sum, dws + dqt::kAbsmeanBlocks, sizeof(double), cudaMemcpyDeviceToHost,
                      st) != cudaSuccess)
    return DQT_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return DQT_ERR_CUDA;
  const double absmean = sum / static_cast<double>(numel);
  if (!dqt::absmean_ok(absmean)) return DQT_ERR_ARG;
  const float s = static_cast<float>(static_cast<double>(grid.qmax) / absmean);
  *s_w = s;
  return dqt::launch_absmean_codes(W0, numel, s, grid.qmin, grid.qmax, codes, st) ? DQT_ERR_CUDA
                                                                                    : DQT_OK;
}

int dqt_act_quant(const dqt_bf16* X, int64_t T, int64_t K, int8_t* Xq, float* s_x,
                  void* stream) {
  if (!X || !Xq || !s_x || T <= 0 || K <= 0) return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim) return DQT_ERR_RANGE;
  if (K % 8 || !aligned16(X) || (reinterpret_cast<uintptr_t>(Xq) & 7u)) return DQT_ERR_ALIGN;
  return dqt::launch_act_quant(X, T, K, Xq, s_x, nullptr, nullptr, as_stream(stream))
             ? DQT_ERR_CUDA
             : DQT_OK;
}

int dqt_act_quant_images(const dqt_bf16* X, int64_t T, int64_t K, int8_t* Xq, float* s_x,
                         dqt_bf16* Xq_img, dqt_bf16* Xdq, void* stream) {
  if (!X || !s_x || (!Xq && !Xq_img && !Xdq) || T <= 0 || K <= 0) return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim) return DQT_ERR_RANGE;
  if (K % 8 || !aligned16(X) || (Xq && (reinterpret_cast<uintptr_t>(Xq) & 7u)) ||
      (Xq_img && !aligned16(Xq_img)) || (Xdq && !aligned16(Xdq)))
    return DQT_ERR_ALIGN;
  return dqt::launch_act_quant(X, T, K, Xq, s_x, Xq_img, Xdq, as_stream(stream)) ? DQT_ERR_CUDA
                                                                                 : DQT_OK;
}

int dqt_codes_to_xdq(const int8_t* Xq, const float* s_x, int64_t T, int64_t K, dqt_bf16* Xdq,
                     void* stream) {
  if (!Xq || !s_x || !Xdq || T <= 0 || K <= 0) return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim) return DQT_ERR_RANGE;
  if (K % 16 || !aligned16(Xq) || !aligned16(Xdq)) return DQT_ERR_ALIGN;
  return dqt::launch_codes_to_xdq(Xq, s_x, T, K, Xdq, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_codes_to_bf16(const int8_t* W, int64_t numel, dqt_bf16* W_img, void* stream) {
  if (!W || !W_img || numel <= 0) return DQT_ERR_ARG;
  if (!aligned16(W) || !aligned16(W_img)) return DQT_ERR_ALIGN;
  return dqt::launch_codes_to_bf16(W, numel, W_img, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_rope_bf16(const dqt_bf16* x, dqt_bf16* y, const float* cos_sin, int64_t rows, int64_t S,
                  int64_t H, int64_t D, int32_t inverse, void* stream) {
  if (!x || !y || !cos_sin || rows <= 0 || S <= 0 || H <= 0 || D <= 0) return DQT_ERR_ARG;
  if (inverse != 0 && inverse != 1) return DQT_ERR_ARG;
  if (D % 8 != 0 || !aligned16(x) || !aligned16(y) || !aligned16(cos_sin)) return DQT_ERR_ALIGN;
  if (rows > kMaxDim || S > kMaxDim || H > kMaxDim || D > kMaxDim || H * D > kMaxDim)
    return DQT_ERR_RANGE;
  return dqt::launch_rope(x, y, cos_sin, rows, S, H, D, inverse == 1, as_stream(stream))
             ? DQT_ERR_CUDA
             : DQT_OK;
}

int dqt_cross_entropy_fwd_bf16(const dqt_bf16* logits, const int64_t* targets, int64_t M,
                               int64_t V, float* lse, float* row_loss, void* stream) {
  if (!logits || !targets || !lse || !row_loss || M <= 0 || V <= 0) return DQT_ERR_ARG;
  if (V % 8 != 0 || !aligned16(logits)) return DQT_ERR_ALIGN;
  if (M > kMaxDim || V > kMaxDim) return DQT_ERR_RANGE;
  return dqt::launch_ce_fwd(logits, targets, M, V, lse, row_loss, as_stream(stream))
             ? DQT_ERR_CUDA
             : DQT_OK;
}

int dqt_cross_entropy_bwd_bf16(const dqt_bf16* logits, const int64_t* targets, const float* lse,
                               const float* scale, int64_t M, int64_t V, dqt_bf16* dlogits,
                               void* stream) {
  if (!logits || !targets || !lse || !scale || !dlogits || M <= 0 || V <= 0) return DQT_ERR_ARG;
  if (V % 8 != 0 || !aligned16(logits) || !aligned16(dlogits)) return DQT_ERR_ALIGN;
  if (M > kMaxDim || V > kMaxDim) return DQT_ERR_RANGE;
  return dqt::launch_ce_bwd(logits, targets, lse, scale, M, V, dlogits, as_stream(stream))
             ? DQT_ERR_CUDA
             : DQT_OK;
}

int dqt_swiglu_bf16(const dqt_bf16* g, const dqt_bf16* u, dqt_bf16* h, int64_t n, void* stream) {
  if (!g || !u || !h || n <= 0) return DQT_ERR_ARG;
  if (n % 8 != 0 || !aligned16(g) || !aligned16(u) || !aligned16(h)) return DQT_ERR_ALIGN;
  return dqt::launch_swiglu(g, u, h, n, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_swiglu_bwd_bf16(const dqt_bf16* g, const dqt_bf16* u, const dqt_bf16* dh, dqt_bf16* dg,
                        dqt_bf16* du, int64_t n, void* stream) {
  if (!g || !u || !dh || !dg || !du || n <= 0) return DQT_ERR_ARG;
  if (n % 8 != 0 || !aligned16(g) || !aligned16(u) || !aligned16(dh) || !aligned16(dg) ||
      !aligned16(du))
    return DQT_ERR_ALIGN;
  return dqt::launch_swiglu_bwd(g, u, dh, dg, du, n, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_rmsnorm_bf16(const dqt_bf16* x, const dqt_bf16* w, float eps, int64_t rows, int64_t D,
                     dqt_bf16* y, float* rstd, void* stream) {
  if (!x || !w || !y || !rstd || rows <= 0 || D <= 0 || !(eps >= 0.0f)) return DQT_ERR_ARG;
  if (D % 8 != 0 || !aligned16(x) || !aligned16(w) || !aligned16(y)) return DQT_ERR_ALIGN;
  if (D > 2048 || rows > kMaxDim) return DQT_ERR_RANGE;
  return dqt::launch_rmsnorm(x, w, eps, rows, D, y, rstd, as_stream(stream)) ? DQT_ERR_CUDA
                                                                              : DQT_OK;
}

size_t dqt_rmsnorm_bwd_workspace_size(int64_t rows, int64_t D) {
  if (rows <= 0 || D <= 0 || D > 2048 || rows > kMaxDim) return 0;
  return dqt::rmsnorm_bwd_ws(rows, D);
}

int dqt_rmsnorm_bwd_bf16(const dqt_bf16* x, const dqt_bf16* w, const float* rstd,
                         const dqt_bf16* dy, int64_t rows, int64_t D, dqt_bf16* dx, dqt_bf16* dw,
                         void* ws, size_t ws_bytes, void* stream) {
  if (!x || !w || !rstd || !dy || !dx || !dw || !ws || rows <= 0 || D <= 0) return DQT_ERR_ARG;
  if (D % 8 != 0 || !aligned16(x) || !aligned16(w) || !aligned16(dy) || !aligned16(dx) ||
      !aligned16(ws))
    return DQT_ERR_ALIGN;
  if (D > 2048 || rows > kMaxDim) return DQT_ERR_RANGE;
  if (ws_bytes < dqt::rmsnorm_bwd_ws(rows, D)) return DQT_ERR_ARG;
  return dqt::launch_rmsnorm_bwd(x, w, rstd, dy, rows, D, dx, dw, static_cast<float*>(ws),
                                 as_stream(stream))
             ? DQT_ERR_CUDA
             : DQT_OK;
}

// |sum| <= K * 128 * max|c| must fit int32 (checked before any launch).
static bool fwd_range_ok(dqt_grid_t grid, int64_t K) {
  const int64_t cmax = grid.qmax > -grid.qmin ? grid.qmax : -grid.qmin;
  const int64_t cm = cmax > 0 ? cmax : 1;
  return K * 128 * cm <= (int64_t(1) << 31) - 1;
}

// The exact integer forward (both operand forms): the reduction is cut into
// chunks whose partial sums stay <= 2^24 (exact in fp32).
static int fwd_launch(const void* A, const float* s_x, const void* B, float s_w,
               dqt_grid_t grid, int64_t T, int64_t K, int64_t N, dqt_bf16* Y, int32_t* acc_out,
               void* tail_ws, size_t tail_bytes, void* stream, int split = 0,
               float s_w1 = 0.0f) {
  const int64_t cmax = grid.qmax > -grid.qmin ? grid.qmax : -grid.qmin;
  const int64_t cm = cmax > 0 ? cmax : 1;
  // Largest chunk whose partial sums stay <= 2^24 (exact in fp32), multiple of 64.
  int64_t chunk = ((int64_t(1) << 24) / (128 * cm)) / 64 * 64;
  if (chunk < 64) chunk = 64;
  if (chunk > kMaxDim) chunk = int64_t(1) << 30;
  dqt::GemmLaunch g{};
  g.kind = dqt::GEMM_FWD;
  g.M = static_cast<int>(T);
  g.N = static_cast<int>(N);
  g.Kred = static_cast<int>(K);
  g.A = A;
  g.B = B;
  g.chunk_k = static_cast<int>(chunk);
  g.s_x = s_x;
  g.scale = s_w;
  g.out_bf16 = Y;
  g.acc_out = acc_out;
  g.ws = tail_ws;
  g.ws_bytes = tail_ws ? tail_bytes : 0;
  g.split = split;
  g.scale1 = s_w1;
  return dqt::launch_gemm(g, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

static inline size_t fwd_ws_align(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// Workspace of the last-wave reduction slices of a 2-SM forward or dX GEMM
// (M x N output reduced over Kred); 0 with 1-SM tiles.
static size_t gemm_tail_ws(int64_t M, int64_t N, int64_t Kred) {
  if (dqt::gemm_mode() != 0) return 0;
  return dqt::gemm_tail_bytes(static_cast<int>(M), static_cast<int>(N), static_cast<int>(Kred));
}

size_t dqt_fwd_workspace_size(int64_t T, int64_t K, int64_t N) {
  if (T <= 0 || K <= 0 || N <= 0 || T > kMaxDim || K > kMaxDim || N > kMaxDim) return 0;
  return fwd_ws_align(static_cast<size_t>(T) * static_cast<size_t>(K) * 2u) +
         fwd_ws_align(static_cast<size_t>(N) * static_cast<size_t>(K) * 2u) +
         dqt_fwd_img_workspace_size(T, K, N);
}

size_t dqt_fwd_img_workspace_size(int64_t T, int64_t K, int64_t N) {
  if (T <= 0 || K <= 0 || N <= 0 || T > kMaxDim || K > kMaxDim || N > kMaxDim) return 0;
  return gemm_tail_ws(T, N, K);
}

int dqt_bitlinear_fwd(const int8_t* Xq, const float* s_x, const int8_t* W, float s_w,
                      dqt_grid_t grid, int64_t T, int64_t K, int64_t N, dqt_bf16* Y,
                      int32_t* acc_out, void* ws, size_t ws_bytes, void* stream) {
  if (!Xq || !s_x || !W || !Y || !ws || T <= 0 || K <= 0 || N <= 0 || !grid_ok(grid) ||
      !(s_w > 0.0f) || !isfinite(s_w))
    return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim || !fwd_range_ok(grid, K)) return DQT_ERR_RANGE;
  if (ws_bytes < dqt_fwd_workspace_size(T, K, N)) return DQT_ERR_ARG;
  if (K % 8 || N % 8 || !aligned16(Xq) || !aligned16(W) || !aligned16(Y) || !aligned16(ws) ||
      (acc_out && !aligned16(acc_out)))
    return DQT_ERR_ALIGN;
  // the exact bf16 images of both operands' codes, then the GEMM on them
  cudaStream_t st = as_stream(stream);
  const size_t x_bytes = fwd_ws_align(static_cast<size_t>(T) * static_cast<size_t>(K) * 2u);
  const size_t w_bytes = fwd_ws_align(static_cast<size_t>(N) * static_cast<size_t>(K) * 2u);
  dqt_bf16* Xq_img = static_cast<dqt_bf16*>(ws);
  dqt_bf16* W_img = reinterpret_cast<dqt_bf16*>(static_cast<uint8_t*>(ws) + x_bytes);
  if (dqt::launch_codes_to_bf16(Xq, T * K, Xq_img, st) ||
      dqt::launch_codes_to_bf16(W, N * K, W_img, st))
    return DQT_ERR_CUDA;
  return fwd_launch(Xq_img, s_x, W_img, s_w, grid, T, K, N, Y, acc_out,
                    static_cast<uint8_t*>(ws) + x_bytes + w_bytes, ws_bytes - x_bytes - w_bytes,
                    stream);
}

int dqt_bitlinear_fwd_img(const dqt_bf16* Xq_img, const float* s_x, const dqt_bf16* W_img,
                          float s_w, dqt_grid_t grid, int64_t T, int64_t K, int64_t N,
                          dqt_bf16* Y, int32_t* acc_out, void* ws, size_t ws_bytes,
                          void* stream) {
  if (!Xq_img || !s_x || !W_img || !Y || T <= 0 || K <= 0 || N <= 0 || !grid_ok(grid) ||
      !(s_w > 0.0f) || !isfinite(s_w))
    return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim) return DQT_ERR_RANGE;
  if (ws && ws_bytes < dqt_fwd_img_workspace_size(T, K, N)) return DQT_ERR_ARG;
  if (K % 8 || N % 8 || !aligned16(Xq_img) || !aligned16(W_img) || !aligned16(Y) ||
      (acc_out && !aligned16(acc_out)) || (ws && !aligned16(ws)))
    return DQT_ERR_ALIGN;
  if (!fwd_range_ok(grid, K)) return DQT_ERR_RANGE;
  return fwd_launch(Xq_img, s_x, W_img, s_w, grid, T, K, N, Y, acc_out, ws, ws_bytes, stream);
}

// Two weights stacked along N that read the same input (rows [0, N0) the
// first weight's codes with scale s_w0, rows [N0, N) the second's with s_w1).
static bool pair_split_ok(int64_t N0, int64_t N) { return N0 > 0 && N0 < N && N0 % 256 == 0; }

int dqt_bitlinear_fwd_img_pair(const dqt_bf16* Xq_img, const float* s_x, const dqt_bf16* W_img,
                               int64_t N0, float s_w0, float s_w1, dqt_grid_t grid, int64_t T,
                               int64_t K, int64_t N, dqt_bf16* Y, int32_t* acc_out, void* ws,
                               size_t ws_bytes, void* stream) {
  if (!Xq_img || !s_x || !W_img || !Y || T <= 0 || K <= 0 || N <= 0 || !grid_ok(grid) ||
      !(s_w0 > 0.0f) || !isfinite(s_w0) || !(s_w1 > 0.0f) || !isfinite(s_w1) ||
      !pair_split_ok(N0, N))
    return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim) return DQT_ERR_RANGE;
  if (ws && ws_bytes < dqt_fwd_img_workspace_size(T, K, N)) return DQT_ERR_ARG;
  if (K % 8 || N % 8 || !aligned16(Xq_img) || !aligned16(W_img) || !aligned16(Y) ||
      (acc_out && !aligned16(acc_out)) || (ws && !aligned16(ws)))
    return DQT_ERR_ALIGN;
  if (!fwd_range_ok(grid, K)) return DQT_ERR_RANGE;
  return fwd_launch(Xq_img, s_x, W_img, s_w0, grid, T, K, N, Y, acc_out, ws, ws_bytes, stream,
                    static_cast<int>(N0), s_w1);
}

int dqt_act_quant_fp8(const dqt_bf16* X, int64_t T, int64_t K, uint8_t* Xq8, float* s_x8,
                      dqt_bf16* Xdq, void* stream) {
  if (!X || !Xq8 || !s_x8 || T <= 0 || K <= 0) return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim) return DQT_ERR_RANGE;
  if (K % 16 || !aligned16(X) || !aligned16(Xq8) || (Xdq && !aligned16(Xdq)))
    return DQT_ERR_ALIGN;
  return dqt::launch_act_quant_fp8(X, T, K, Xq8, s_x8, Xdq, as_stream(stream)) ? DQT_ERR_CUDA
                                                                              : DQT_OK;
}

int dqt_codes_to_fp8(const int8_t* W, int64_t numel, dqt_grid_t grid, uint8_t* W8, void* stream) {
  if (!W || !W8 || numel <= 0 || !grid_ok(grid)) return DQT_ERR_ARG;
  if (grid.qmin < -16 || grid.qmax > 16) return DQT_ERR_RANGE;
  if (!aligned16(W) || !aligned16(W8)) return DQT_ERR_ALIGN;
  return dqt::launch_codes_to_fp8(W, numel, W8, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_codes_to_fp8_split(const int8_t* W, int64_t N, int64_t K, uint8_t* W8, void* stream) {
  if (!W || !W8 || N <= 0 || K <= 0) return DQT_ERR_ARG;
  if (N > kMaxDim || K > kMaxDim) return DQT_ERR_RANGE;
  if (K % 16 || !aligned16(W) || !aligned16(W8)) return DQT_ERR_ALIGN;
  return dqt::launch_codes_to_fp8_split(W, N, K, W8, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

// The E4M3 forward's weight form for a grid: codes within 16 in magnitude are
// E4M3 values (W8 [N, K]); wider codes take the split image (W8 [N, 2K], the
// activation row read for both halves; K a multiple of 128).
static bool fp8_split(dqt_grid_t grid) { return grid.qmin < -16 || grid.qmax > 16; }

int dqt_bitlinear_fwd_fp8(const uint8_t* Xq8, const float* s_x8, const uint8_t* W8, float s_w,
                          dqt_grid_t grid, int64_t T, int64_t K, int64_t N, dqt_bf16* Y,
                          float* acc_out, void* stream) {
  if (!Xq8 || !s_x8 || !W8 || !Y || T <= 0 || K <= 0 || N <= 0 || !grid_ok(grid) ||
      !(s_w > 0.0f) || !isfinite(s_w))
    return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim) return DQT_ERR_RANGE;
  const bool split = fp8_split(grid);
  if (K % (split ? 128 : 16) || N % 8 || !aligned16(Xq8) || !aligned16(W8) || !aligned16(Y) ||
      (acc_out && !aligned16(acc_out)))
    return DQT_ERR_ALIGN;
  dqt::GemmLaunch g{};
  g.kind = dqt::GEMM_FWD8;
  g.M = static_cast<int>(T);
  g.N = static_cast<int>(N);
  g.Kred = static_cast<int>(split ? 2 * K : K);
  g.a_wrap = split ? static_cast<int>(K) : 0;
  g.A = Xq8;
  g.B = W8;
  g.pair = true;
  g.s_x = s_x8;
  g.scale = s_w;
  g.out_bf16 = Y;
  g.acc_f32 = acc_out;
  return dqt::launch_gemm(g, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_bitlinear_fwd_fp8_pair(const uint8_t* Xq8, const float* s_x8, const uint8_t* W8, int64_t N0,
                               float s_w0, float s_w1, dqt_grid_t grid, int64_t T, int64_t K,
                               int64_t N, dqt_bf16* Y, float* acc_out, void* stream) {
  if (!Xq8 || !s_x8 || !W8 || !Y || T <= 0 || K <= 0 || N <= 0 || !grid_ok(grid) ||
      !(s_w0 > 0.0f) || !isfinite(s_w0) || !(s_w1 > 0.0f) || !isfinite(s_w1) ||
      !pair_split_ok(N0, N))
    return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim) return DQT_ERR_RANGE;
  const bool split = fp8_split(grid);
  if (K % (split ? 128 : 16) || N % 8 || !aligned16(Xq8) || !aligned16(W8) || !aligned16(Y) ||
      (acc_out && !aligned16(acc_out)))
    return DQT_ERR_ALIGN;
  dqt::GemmLaunch g{};
  g.kind = dqt::GEMM_FWD8;
  g.M = static_cast<int>(T);
  g.N = static_cast<int>(N);
  g.Kred = static_cast<int>(split ? 2 * K : K);
  g.a_wrap = split ? static_cast<int>(K) : 0;
  g.A = Xq8;
  g.B = W8;
  g.pair = true;
  g.s_x = s_x8;
  g.scale = s_w0;
  g.split = static_cast<int>(N0);
  g.scale1 = s_w1;
  g.out_bf16 = Y;
  g.acc_f32 = acc_out;
  return dqt::launch_gemm(g, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

static inline size_t ws_align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

size_t dqt_bwd_dx_workspace_size(int64_t T, int64_t N, int64_t K) {
  if (T <= 0 || N <= 0 || K <= 0 || T > kMaxDim || N > kMaxDim || K > kMaxDim) return 0;
  return ws_align256(static_cast<size_t>(N) * static_cast<size_t>(K) * 2u) +
         dqt_bwd_dx_img_workspace_size(T, N, K);
}

size_t dqt_bwd_dx_img_workspace_size(int64_t T, int64_t N, int64_t K) {
  if (T <= 0 || N <= 0 || K <= 0 || T > kMaxDim || N > kMaxDim || K > kMaxDim) return 0;
  return gemm_tail_ws(T, K, N);
}

int dqt_bitlinear_bwd_dx(const dqt_bf16* dY, const int8_t* W, float s_w, int64_t T, int64_t N,
                         int64_t K, dqt_bf16* dX, void* ws, size_t ws_bytes, void* stream) {
  if (!dY || !W || !dX || !ws || T <= 0 || N <= 0 || K <= 0 || !(s_w > 0.0f) || !isfinite(s_w))
    return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim) return DQT_ERR_RANGE;
  if (ws_bytes < dqt_bwd_dx_workspace_size(T, N, K)) return DQT_ERR_ARG;
  if (K % 8 || N % 8 || !aligned16(dY) || !aligned16(W) || !aligned16(dX) || !aligned16(ws))
    return DQT_ERR_ALIGN;
  // the exact bf16 image of the codes, then the GEMM on it (the rest of the
  // workspace holds its last-wave slice partials)
  const size_t w_bytes = ws_align256(static_cast<size_t>(N) * static_cast<size_t>(K) * 2u);
  dqt_bf16* W_img = static_cast<dqt_bf16*>(ws);
  if (dqt::launch_codes_to_bf16(W, N * K, W_img, as_stream(stream))) return DQT_ERR_CUDA;
  return dqt_bitlinear_bwd_dx_img(dY, W_img, s_w, T, N, K, dX, static_cast<uint8_t*>(ws) + w_bytes,
                                  ws_bytes - w_bytes, stream);
}

int dqt_bitlinear_bwd_dx_img(const dqt_bf16* dY, const dqt_bf16* W_img, float s_w, int64_t T,
                             int64_t N, int64_t K, dqt_bf16* dX, void* ws, size_t ws_bytes,
                             void* stream) {
  return dqt_bitlinear_bwd_dx_img_ld(dY, N, W_img, s_w, T, N, K, dX, ws, ws_bytes, stream);
}

int dqt_bitlinear_bwd_dx_img_ld(const dqt_bf16* dY, int64_t ldy, const dqt_bf16* W_img, float s_w,
                                int64_t T, int64_t N, int64_t K, dqt_bf16* dX, void* ws,
                                size_t ws_bytes, void* stream) {
  if (!dY || !W_img || !dX || T <= 0 || N <= 0 || K <= 0 || !(s_w > 0.0f) || !isfinite(s_w) ||
      ldy < N)
    return DQT_ERR_ARG;
  if (ldy > kMaxDim) return DQT_ERR_RANGE;
  if (ldy % 8) return DQT_ERR_ALIGN;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim) return DQT_ERR_RANGE;
  if (ws && ws_bytes < dqt_bwd_dx_img_workspace_size(T, N, K)) return DQT_ERR_ARG;
  if (K % 8 || N % 8 || !aligned16(dY) || !aligned16(W_img) || !aligned16(dX) ||
      (ws && !aligned16(ws)))
    return DQT_ERR_ALIGN;
  dqt::GemmLaunch g{};
  g.kind = dqt::GEMM_DX;
  g.M = static_cast<int>(T);
  g.N = static_cast<int>(K);
  g.Kred = static_cast<int>(N);
  g.A = dY;
  g.B = W_img;
  g.scale = 1.0f / s_w;
  g.out_bf16 = dX;
  g.ws = ws;
  g.ws_bytes = ws ? ws_bytes : 0;
  g.lda = ldy;
  return dqt::launch_gemm(g, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

size_t dqt_bwd_dw_workspace_size(int64_t T, int64_t N, int64_t K) {
  if (T <= 0 || N <= 0 || K <= 0 || T > kMaxDim || N > kMaxDim || K > kMaxDim) return 0;
  return ws_align256(static_cast<size_t>(T) * static_cast<size_t>(K) * 2u) +
         dqt_bwd_dw_img_workspace_size(T, N, K);
}

size_t dqt_bwd_dw_img_workspace_size(int64_t T, int64_t N, int64_t K) {
  if (T <= 0 || N <= 0 || K <= 0 || T > kMaxDim || N > kMaxDim || K > kMaxDim) return 0;
  if (dqt::gemm_mode() != 0) return 0;
  const int s = dqt::dw_splits(static_cast<int>(N), static_cast<int>(K), static_cast<int>(T));
  if (s > 1) return static_cast<size_t>(s) * static_cast<size_t>(N) * static_cast<size_t>(K) * 4u;
  // last-wave tail: at most one 256 x 256 fp32 slice partial per cluster (at
  // most one cluster per SM pair on any launch)
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const dqt::TailPlan tp =
      dqt::tail_plan(static_cast<int>(N), static_cast<int>(K), static_cast<int>(T), sms / 2);
  if (tp.splits < 2) return 0;
  return 256 + static_cast<size_t>(sms / 2) * 65536 * sizeof(float);  // + 256: alignment
}

int dqt_bitlinear_bwd_dw_update(const dqt_bf16* dY, const int8_t* Xq, const float* s_x,
                                int8_t* W, float s_w, float* m, float* v, const dqt_adamw_t* hp,
                                const dqt_sr_t* sr, dqt_grid_t grid, int64_t T, int64_t N,
                                int64_t K, float* dW_out, unsigned long long* changed_out,
                                void* ws, size_t ws_bytes, void* stream) {
  if (!dY || !Xq || !s_x || !ws || T <= 0 || N <= 0 || K <= 0) return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim || N * K > (int64_t(1) << 62)) return DQT_ERR_RANGE;
  const size_t img = ws_align256(static_cast<size_t>(T) * static_cast<size_t>(K) * 2u);
  if (ws_bytes < img) return DQT_ERR_ARG;
  if (K % 16 || N % 8 || !aligned16(Xq) || !aligned16(ws) || !aligned16(dY) ||
      (W && !aligned16(W)) || (m && !aligned16(m)) || (v && !aligned16(v)) ||
      (dW_out && !aligned16(dW_out)))
    return DQT_ERR_ALIGN;
  // the argument checks of the GEMM call before anything is launched
  const bool upd = W || m || v;
  if (upd && (!W || !m || !v)) return DQT_ERR_ARG;
  if (!upd && !dW_out) return DQT_ERR_ARG;
  if (upd) {
    dqt::UpdateConsts uc;
    const int rc = make_update_consts(hp, sr, grid, s_w, &uc);
    if (rc != DQT_OK) return rc;
  }
  // X_tilde = bf16(q / s_x) into the workspace, then the GEMM + update on it;
  // the rest of the workspace serves the token-sliced reduction
  dqt_bf16* Xdq = static_cast<dqt_bf16*>(ws);
  if (dqt::launch_codes_to_xdq(Xq, s_x, T, K, Xdq, as_stream(stream))) return DQT_ERR_CUDA;
  uint8_t* rest = static_cast<uint8_t*>(ws) + img;
  const size_t rest_bytes = ws_bytes - img;
  return dqt_bitlinear_bwd_dw_update_img(dY, Xdq, W, s_w, m, v, hp, sr, grid, T, N, K, dW_out, nullptr,
                                         nullptr, changed_out, rest_bytes ? rest : nullptr, rest_bytes,
                                         stream);
}

int dqt_bitlinear_bwd_dw_update_img(const dqt_bf16* dY, const dqt_bf16* Xdq, int8_t* W,
                                    float s_w, float* m, float* v, const dqt_adamw_t* hp,
                                    const dqt_sr_t* sr, dqt_grid_t grid, int64_t T, int64_t N,
                                    int64_t K, float* dW_out, dqt_bf16* W_img_next,
                                    uint8_t* W8_next, unsigned long long* changed_out, void* ws,
                                    size_t ws_bytes, void* stream) {
  const bool upd = W || m || v;
  if (!dY || !Xdq || T <= 0 || N <= 0 || K <= 0) return DQT_ERR_ARG;
  if (upd && (!W || !m || !v)) return DQT_ERR_ARG;
  if (!upd && (!dW_out || W_img_next || W8_next)) return DQT_ERR_ARG;
  // codes wider than E4M3's exact integers: W8_next receives the split image
  const bool w8_split = W8_next && fp8_split(grid);
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim || N * K > (int64_t(1) << 62)) return DQT_ERR_RANGE;
  if (K % 8 || N % 8 || (w8_split && K % 16) || !aligned16(dY) || !aligned16(Xdq) ||
      (W && !aligned16(W)) ||
      (m && !aligned16(m)) || (v && !aligned16(v)) || (dW_out && !aligned16(dW_out)) ||
      (W_img_next && !aligned16(W_img_next)) || (W8_next && !aligned16(W8_next)) ||
      (ws && !aligned16(ws)))
    return DQT_ERR_ALIGN;
  dqt::GemmLaunch g{};
  g.ws = ws;
  g.ws_bytes = ws ? ws_bytes : 0;
  if (upd) {
    const int rc = make_update_consts(hp, sr, grid, s_w, &g.uc);
    if (rc != DQT_OK) return rc;
  }
  g.kind = dqt::GEMM_DW;
  g.M = static_cast<int>(N);
  g.N = static_cast<int>(K);
  g.Kred = static_cast<int>(T);
  g.A = dY;
  g.B = Xdq;
  g.W = upd ? W : nullptr;
  g.m = m;
  g.v = v;
  g.dW_out = dW_out;
  g.img_next = W_img_next;
  g.img8_next = W8_next;
  g.img8_split = w8_split;
  g.changed = upd ? changed_out : nullptr;
  return dqt::launch_gemm(g, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_bitlinear_bwd_dw_update_img_pair(const dqt_bf16* dY, const dqt_bf16* Xdq, int8_t* W,
                                         int64_t N0, float s_w0, float s_w1, float* m, float* v,
                                         const dqt_adamw_t* hp, const dqt_sr_t* sr0,
                                         const dqt_sr_t* sr1, dqt_grid_t grid, int64_t T,
                                         int64_t N, int64_t K, float* dW_out,
                                         dqt_bf16* W_img_next, uint8_t* W8_next,
                                         unsigned long long* changed_out, void* ws,
                                         size_t ws_bytes, void* stream) {
  if (!dY || !Xdq || !W || !m || !v || T <= 0 || N <= 0 || K <= 0 || !pair_split_ok(N0, N))
    return DQT_ERR_ARG;
  const bool w8_split = W8_next && fp8_split(grid);
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim || N * K > (int64_t(1) << 62)) return DQT_ERR_RANGE;
  if (K % 8 || N % 8 || (w8_split && K % 16) || !aligned16(dY) || !aligned16(Xdq) ||
      !aligned16(W) || !aligned16(m) ||
      !aligned16(v) || (dW_out && !aligned16(dW_out)) ||
      (W_img_next && !aligned16(W_img_next)) || (W8_next && !aligned16(W8_next)) ||
      (ws && !aligned16(ws)))
    return DQT_ERR_ALIGN;
  dqt::GemmLaunch g{};
  g.ws = ws;
  g.ws_bytes = ws ? ws_bytes : 0;
  int rc = make_update_consts(hp, sr0, grid, s_w0, &g.uc);
  if (rc == DQT_OK) rc = make_update_consts(hp, sr1, grid, s_w1, &g.uc1);
  if (rc != DQT_OK) return rc;
  g.split = static_cast<int>(N0);
  g.kind = dqt::GEMM_DW;
  g.M = static_cast<int>(N);
  g.N = static_cast<int>(K);
  g.Kred = static_cast<int>(T);
  g.A = dY;
  g.B = Xdq;
  g.W = W;
  g.m = m;
  g.v = v;
  g.dW_out = dW_out;
  g.img_next = W_img_next;
  g.img8_next = W8_next;
  g.img8_split = w8_split;
  g.changed = changed_out;
  return dqt::launch_gemm(g, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

// One problem of a grouped call into a launch record (the checks of the
// single and stacked calls).
static int dw_problem(const dqt_dw_problem_t& q, const dqt_adamw_t* hp, dqt_grid_t grid,
                      int64_t T, dqt::GemmLaunch& g) {
  const int64_t N = q.N, K = q.K;
  if (!q.dY || !q.Xdq || !q.W || !q.m || !q.v || !q.sr0 || T <= 0 || N <= 0 || K <= 0)
    return DQT_ERR_ARG;
  if (q.N0 != 0 && (!pair_split_ok(q.N0, N) || !q.sr1)) return DQT_ERR_ARG;
  const bool w8_split = q.W8_next && fp8_split(grid);
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim || N * K > (int64_t(1) << 62)) return DQT_ERR_RANGE;
  if (K % 8 || N % 8 || (w8_split && K % 16) || !aligned16(q.dY) || !aligned16(q.Xdq) ||
      !aligned16(q.W) || !aligned16(q.m) || !aligned16(q.v) ||
      (q.W_img_next && !aligned16(q.W_img_next)) || (q.W8_next && !aligned16(q.W8_next)))
    return DQT_ERR_ALIGN;
  g = dqt::GemmLaunch{};
  int rc = make_update_consts(hp, q.sr0, grid, q.s_w0, &g.uc);
  if (rc == DQT_OK && q.N0 != 0) rc = make_update_consts(hp, q.sr1, grid, q.s_w1, &g.uc1);
  if (rc != DQT_OK) return rc;
  g.split = static_cast<int>(q.N0);
  g.kind = dqt::GEMM_DW;
  g.M = static_cast<int>(N);
  g.N = static_cast<int>(K);
  g.Kred = static_cast<int>(T);
  g.A = q.dY;
  g.B = q.Xdq;
  g.W = q.W;
  g.m = q.m;
  g.v = q.v;
  g.img_next = q.W_img_next;
  g.img8_next = q.W8_next;
  g.img8_split = w8_split;
  g.changed = q.changed_out;
  return DQT_OK;
}

int dqt_bitlinear_bwd_dw_update_group(const dqt_dw_problem_t* probs, int nprob,
                                      const dqt_adamw_t* hp, dqt_grid_t grid, int64_t T,
                                      void* stream) {
  if (!probs || nprob != 2) return DQT_ERR_ARG;
  dqt::GemmLaunch g[2];
  for (int i = 0; i < 2; ++i) {
    const int rc = dw_problem(probs[i], hp, grid, T, g[i]);
    if (rc != DQT_OK) return rc;
  }
  return dqt::launch_dw_group(g[0], g[1], as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_sr_update(const float* grad, int8_t* W, float s_w, float* m, float* v,
                  const dqt_adamw_t* hp, const dqt_sr_t* sr, dqt_grid_t grid, int64_t numel,
                  unsigned long long* changed_out, void* stream) {
  if (!grad || !W || !m || !v || numel <= 0) return DQT_ERR_ARG;
  if (!aligned16(grad) || !aligned16(W) || !aligned16(m) || !aligned16(v)) return DQT_ERR_ALIGN;
  dqt::UpdateConsts uc;
  const int rc = make_update_consts(hp, sr, grid, s_w, &uc);
  if (rc != DQT_OK) return rc;
  return dqt::launch_sr_update(grad, W, m, v, numel, uc, nullptr, changed_out, as_stream(stream))
             ? DQT_ERR_CUDA
             : DQT_OK;
}

size_t dqt_update_consts_size(void) { return sizeof(dqt::UpdateConsts); }

int dqt_update_consts(const dqt_adamw_t* hp, const dqt_sr_t* sr, dqt_grid_t grid, float s_w,
                      void* out, size_t out_bytes) {
  if (!out || out_bytes < sizeof(dqt::UpdateConsts)) return DQT_ERR_ARG;
  dqt::UpdateConsts uc;
  const int rc = make_update_consts(hp, sr, grid, s_w, &uc);
  if (rc != DQT_OK) return rc;
  memcpy(out, &uc, sizeof(uc));
  return DQT_OK;
}

int dqt_bitlinear_bwd_dw_update_dev(const dqt_bf16* dY, const dqt_bf16* Xdq, int8_t* W, float* m,
                                    float* v, const void* consts_dev, int64_t T, int64_t N,
                                    int64_t K, float* dW_out, dqt_bf16* W_img_next,
                                    uint8_t* W8_next, unsigned long long* changed_out, void* ws,
                                    size_t ws_bytes, void* stream) {
  if (!dY || !Xdq || !W || !m || !v || !consts_dev || T <= 0 || N <= 0 || K <= 0)
    return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim) return DQT_ERR_RANGE;
  if (K % 8 || N % 8 || !aligned16(dY) || !aligned16(Xdq) || !aligned16(W) || !aligned16(m) ||
      !aligned16(v) || !aligned16(consts_dev) || (dW_out && !aligned16(dW_out)) ||
      (W_img_next && !aligned16(W_img_next)) || (W8_next && !aligned16(W8_next)) ||
      (ws && !aligned16(ws)))
    return DQT_ERR_ALIGN;
  dqt::GemmLaunch g{};
  g.ws = ws;
  g.ws_bytes = ws ? ws_bytes : 0;
  g.kind = dqt::GEMM_DW;
  g.M = static_cast<int>(N);
  g.N = static_cast<int>(K);
  g.Kred = static_cast<int>(T);
  g.A = dY;
  g.B = Xdq;
  g.W = W;
  g.m = m;
  g.v = v;
  g.dW_out = dW_out;
  g.img_next = W_img_next;
  g.img8_next = W8_next;
  g.changed = changed_out;
  g.uc_dev = static_cast<const dqt::UpdateConsts*>(consts_dev);
  return dqt::launch_gemm(g, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_sr_update_dev(const float* grad, int8_t* W, float* m, float* v, const void* consts_dev,
                      int64_t numel, unsigned long long* changed_out, void* stream) {
  if (!grad || !W || !m || !v || !consts_dev || numel <= 0) return DQT_ERR_ARG;
  if (!aligned16(grad) || !aligned16(W) || !aligned16(m) || !aligned16(v) || !aligned16(consts_dev))
    return DQT_ERR_ALIGN;
  dqt::UpdateConsts unused{};
  return dqt::launch_sr_update(grad, W, m, v, numel, unused,
                               static_cast<const dqt::UpdateConsts*>(consts_dev), changed_out,
                               as_stream(stream))
             ? DQT_ERR_CUDA
             : DQT_OK;
}

// ---- 2-bit packed ternary codes ----------------------------------------------
int dqt_pack_ternary(const int8_t* codes, int64_t numel, uint8_t* packed, void* stream) {
  if (!codes || !packed || numel <= 0) return DQT_ERR_ARG;
  if (!aligned16(codes) || !aligned16(packed)) return DQT_ERR_ALIGN;
  return dqt::launch_pack_ternary(codes, numel, packed, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_unpack_ternary(const uint8_t* packed, int64_t numel, int8_t* codes, void* stream) {
  if (!codes || !packed || numel <= 0) return DQT_ERR_ARG;
  if (!aligned16(codes) || !aligned16(packed)) return DQT_ERR_ALIGN;
  return dqt::launch_unpack_ternary(packed, numel, codes, as_stream(stream)) ? DQT_ERR_CUDA
                                                                             : DQT_OK;
}

int dqt_packed_to_bf16(const uint8_t* packed, int64_t numel, dqt_bf16* W_img, void* stream) {
  if (!packed || !W_img || numel <= 0) return DQT_ERR_ARG;
  if (!aligned16(packed) || !aligned16(W_img)) return DQT_ERR_ALIGN;
  return dqt::launch_packed_to_bf16(packed, numel, W_img, as_stream(stream)) ? DQT_ERR_CUDA
                                                                             : DQT_OK;
}

int dqt_packed_to_fp8(const uint8_t* packed, int64_t numel, uint8_t* W8, void* stream) {
  if (!packed || !W8 || numel <= 0) return DQT_ERR_ARG;
  if (!aligned16(packed) || !aligned16(W8)) return DQT_ERR_ALIGN;
  return dqt::launch_packed_to_fp8(packed, numel, W8, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

int dqt_sr_update_packed(const float* grad, uint8_t* Wp, float s_w, float* m, float* v,
                         const dqt_adamw_t* hp, const dqt_sr_t* sr, int64_t numel,
                         unsigned long long* changed_out, void* stream) {
  if (!grad || !Wp || !m || !v || numel <= 0) return DQT_ERR_ARG;
  if (!aligned16(grad) || !aligned16(Wp) || !aligned16(m) || !aligned16(v)) return DQT_ERR_ALIGN;
  dqt::UpdateConsts uc;
  const dqt_grid_t tern = {-1, 1};
  const int rc = make_update_consts(hp, sr, tern, s_w, &uc);
  if (rc != DQT_OK) return rc;
  return dqt::launch_sr_update(grad, reinterpret_cast<int8_t*>(Wp), m, v, numel, uc, nullptr,
                               changed_out, as_stream(stream), true)
             ? DQT_ERR_CUDA
             : DQT_OK;
}

int dqt_bitlinear_bwd_dw_update_packed(const dqt_bf16* dY, const dqt_bf16* Xdq, uint8_t* Wp,
                                       float s_w, float* m, float* v, const dqt_adamw_t* hp,
                                       const dqt_sr_t* sr, int64_t T, int64_t N, int64_t K,
                                       float* dW_out, unsigned long long* changed_out, void* ws,
                                       size_t ws_bytes, void* stream) {
  if (!dY || !Xdq || !Wp || !m || !v || T <= 0 || N <= 0 || K <= 0) return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim || N * K > (int64_t(1) << 62)) return DQT_ERR_RANGE;
  if (K % 8 || N % 8 || !aligned16(dY) || !aligned16(Xdq) || !aligned16(Wp) || !aligned16(m) ||
      !aligned16(v) || (dW_out && !aligned16(dW_out)) || (ws && !aligned16(ws)))
    return DQT_ERR_ALIGN;
  dqt::GemmLaunch g{};
  const dqt_grid_t tern = {-1, 1};
  const int rc = make_update_consts(hp, sr, tern, s_w, &g.uc);
  if (rc != DQT_OK) return rc;
  g.ws = ws;
  g.ws_bytes = ws ? ws_bytes : 0;
  g.kind = dqt::GEMM_DW;
  g.M = static_cast<int>(N);
  g.N = static_cast<int>(K);
  g.Kred = static_cast<int>(T);
  g.A = dY;
  g.B = Xdq;
  g.W = reinterpret_cast<int8_t*>(Wp);
  g.packed = true;
  g.m = m;
  g.v = v;
  g.dW_out = dW_out;
  g.changed = changed_out;
  return dqt::launch_gemm(g, as_stream(stream)) ? DQT_ERR_CUDA : DQT_OK;
}

// ---- Adafactor ------------------------------------------------------------------
}  // extern "C"

namespace {

int make_adafactor_consts(const dqt_adafactor_t* hp, dqt::AdafactorConsts* h) {
  if (!hp || hp->step < 1 || !(hp->lr >= 0.0f) || !(hp->eps1 >= 0.0f) || !(hp->eps2 >= 0.0f) ||
      !(hp->clip_d > 0.0f) || !(hp->decay_rate <= 0.0f) || !isfinite(hp->weight_decay) ||
      !isfinite(hp->lr))
    return DQT_ERR_ARG;
  const double t = static_cast<double>(hp->step);
  const double p = pow(t, static_cast<double>(hp->decay_rate));
  h->b2 = static_cast<float>(1.0 - p);
  h->omb2 = static_cast<float>(p);
  if (hp->relative_step) {
    const double cap = hp->warmup_init ? 1e-6 * t : 1e-2;
    const double inv = 1.0 / sqrt(t);
    h->rho = static_cast<float>(cap < inv ? cap : inv);
  } else {
    h->rho = hp->lr;
  }
  h->eps1 = hp->eps1;
  h->eps2 = hp->eps2;
  h->clip_d = hp->clip_d;
  h->weight_decay = hp->weight_decay;
  h->scale_parameter = hp->scale_parameter ? 1 : 0;
  return DQT_OK;
}

int apply_consts(int64_t step_t, const dqt_sr_t* sr, dqt_grid_t grid, dqt::UpdateConsts* uc) {
  if (!sr || step_t < 1 || !grid_ok(grid)) return DQT_ERR_ARG;
  if (sr->round_mode != 0 && sr->round_mode != 1) return DQT_ERR_ARG;
  if (sr->elem0 != 0) return DQT_ERR_ARG;  // the statistics span the whole matrix
  *uc = dqt::UpdateConsts{};
  uc->qmin = grid.qmin;
  uc->qmax = grid.qmax;
  uc->step_lo = static_cast<uint32_t>(step_t);
  uc->tensor_id = sr->tensor_id;
  uc->key0 = static_cast<uint32_t>(sr->seed);
  uc->key1 = static_cast<uint32_t>(sr->seed >> 32);
  uc->round_mode = sr->round_mode;
  return DQT_OK;
}

inline size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

}  // namespace

extern "C" {

size_t dqt_adafactor_workspace_size(int64_t N, int64_t K) {
  if (N <= 0 || K <= 0 || N > kMaxDim || K > kMaxDim) return 0;
  return dqt::adafactor_stats_ws(N, K);
}

int dqt_adafactor_stats(const float* G, const void* W, int32_t packed, float s_w, float* R,
                        float* C, const dqt_adafactor_t* hp, int64_t N, int64_t K, float* a_out,
                        float* b_out, float* scalars_out, void* ws, size_t ws_bytes,
                        void* stream) {
  if (!G || !W || !R || !C || !a_out || !b_out || !scalars_out || !ws || N <= 0 || K <= 0 ||
      !(s_w > 0.0f) || !isfinite(s_w))
    return DQT_ERR_ARG;
  if (N > kMaxDim || K > kMaxDim || N * K > (int64_t(1) << 62)) return DQT_ERR_RANGE;
  if (ws_bytes < dqt::adafactor_stats_ws(N, K)) return DQT_ERR_ARG;
  if (K % 4 || !aligned16(G) || !aligned16(W) || !aligned16(R) || !aligned16(C) ||
      !aligned16(a_out) || !aligned16(b_out) || !aligned16(scalars_out) ||
      (reinterpret_cast<uintptr_t>(ws) & 255u))
    return DQT_ERR_ALIGN;
  dqt::AdafactorConsts h;
  const int rc = make_adafactor_consts(hp, &h);
  if (rc != DQT_OK) return rc;
  return dqt::launch_adafactor_stats(G, static_cast<const int8_t*>(W), packed != 0, s_w, R, C, h,
                                     N, K, ws, a_out, b_out, scalars_out, as_stream(stream))
             ? DQT_ERR_CUDA
             : DQT_OK;
}

int dqt_adafactor_apply(const float* G, void* W, int32_t packed, const float* a, const float* b,
                        const float* scalars, int64_t step_t, const dqt_sr_t* sr, dqt_grid_t grid,
                        int64_t N, int64_t K, unsigned long long* changed_out, void* stream) {
  if (!G || !W || !a || !b || !scalars || N <= 0 || K <= 0) return DQT_ERR_ARG;
  if (N > kMaxDim || K > kMaxDim || N * K > (int64_t(1) << 62)) return DQT_ERR_RANGE;
  if (packed && (grid.qmin != -1 || grid.qmax != 1)) return DQT_ERR_ARG;
  if (K % 4 || !aligned16(G) || !aligned16(W) || !aligned16(a) || !aligned16(b) ||
      !aligned16(scalars))
    return DQT_ERR_ALIGN;
  dqt::UpdateConsts uc;
  const int rc = apply_consts(step_t, sr, grid, &uc);
  if (rc != DQT_OK) return rc;
  return dqt::launch_adafactor_apply(G, static_cast<int8_t*>(W), packed != 0, a, b, scalars, uc,
                                     N, K, changed_out, as_stream(stream))
             ? DQT_ERR_CUDA
             : DQT_OK;
}

size_t dqt_bwd_dw_adafactor_workspace_size(int64_t T, int64_t N, int64_t K) {
  if (T <= 0 || N <= 0 || K <= 0 || T > kMaxDim || N > kMaxDim || K > kMaxDim) return 0;
  const size_t g = align256(static_cast<size_t>(N) * static_cast<size_t>(K) * 4u);
  const size_t st = align256(dqt::adafactor_stats_ws(N, K));
  return g + st + align256(dqt_bwd_dw_img_workspace_size(T, N, K));
}

int dqt_bitlinear_bwd_dw_adafactor(const dqt_bf16* dY, const dqt_bf16* Xdq, void* W,
                                   int32_t packed, float s_w, float* R, float* C,
                                   const dqt_adafactor_t* hp, const dqt_sr_t* sr, dqt_grid_t grid,
                                   int64_t T, int64_t N, int64_t K,
                                   unsigned long long* changed_out, void* ws, size_t ws_bytes,
                                   void* stream) {
  if (!dY || !Xdq || !W || !R || !C || !ws || T <= 0 || N <= 0 || K <= 0 || !(s_w > 0.0f) ||
      !isfinite(s_w))
    return DQT_ERR_ARG;
  if (T > kMaxDim || K > kMaxDim || N > kMaxDim || N * K > (int64_t(1) << 62)) return DQT_ERR_RANGE;
  if (packed && (grid.qmin != -1 || grid.qmax != 1)) return DQT_ERR_ARG;
  if (ws_bytes < dqt_bwd_dw_adafactor_workspace_size(T, N, K)) return DQT_ERR_ARG;
  if (K % 8 || N % 8 || !aligned16(dY) || !aligned16(Xdq) || !aligned16(W) || !aligned16(R) ||
      !aligned16(C) || (reinterpret_cast<uintptr_t>(ws) & 255u))
    return DQT_ERR_ALIGN;
  dqt::AdafactorConsts h;
  int rc = make_adafactor_consts(hp, &h);
  if (rc != DQT_OK) return rc;
  dqt::UpdateConsts uc;
  rc = apply_consts(hp->step, sr, grid, &uc);
  if (rc != DQT_OK) return rc;
  uint8_t* base = static_cast<uint8_t*>(ws);
  float* G = reinterpret_cast<float*>(base);
  const size_t g_bytes = align256(static_cast<size_t>(N) * static_cast<size_t>(K) * 4u);
  void* st_ws = base + g_bytes;
  const size_t st_bytes = align256(dqt::adafactor_stats_ws(N, K));
  void* split_ws = base + g_bytes + st_bytes;
  const size_t split_bytes = ws_bytes - g_bytes - st_bytes;
  cudaStream_t s = as_stream(stream);
  // 1. the weight gradient (gradient-only GEMM) into the workspace
  dqt::GemmLaunch g{};
  g.kind = dqt::GEMM_DW;
  g.M = static_cast<int>(N);
  g.N = static_cast<int>(K);
  g.Kred = static_cast<int>(T);
  g.A = dY;
  g.B = Xdq;
  g.dW_out = G;
  g.ws = split_bytes ? split_ws : nullptr;
  g.ws_bytes = split_bytes;
  if (dqt::launch_gemm(g, s)) return DQT_ERR_CUDA;
  // 2. statistics, 3. the per-element step
  const dqt::AdafactorBufs fb = dqt::adafactor_bufs(st_ws, N, K);
  if (dqt::launch_adafactor_stats(G, static_cast<const int8_t*>(W), packed != 0, s_w, R, C, h, N,
                                  K, st_ws, fb.a, fb.b, fb.scalars, s))
    return DQT_ERR_CUDA;
  return dqt::launch_adafactor_apply(G, static_cast<int8_t*>(W), packed != 0, fb.a, fb.b,
                                     fb.scalars, uc, N, K, changed_out, s)
             ? DQT_ERR_CUDA
             : DQT_OK;
}

}  // extern "C"

// Adafactor with stochastic rounding for DQT weights (Sec. 4.3: DQT trained
// with the memory-efficient Adafactor optimiser; Adafactor is Shazeer & Stern,
// ICML 2018).  The second moment of an N x K gradient G is kept factored as
// its row means R [N] and column means C [K]; there is no first moment and no
// per-weight optimiser state, so a step reads G and the codes and writes the
// codes.  Four passes, each HBM-bound or tiny:
//
//   af_sq_partials  one read of G (and the codes): per 128-column chunk row
//                   sums and per 32-row slab column sums of g^2 + eps1, and the
//                   sum of c^2 (for the parameter RMS), in a fixed order
//   af_moments      R <- b2 R + (1 - b2) mean_k, C <- b2 C + (1 - b2) mean_n
//   af_usq_partials second read of G: sum of g^2 / (R[n] C[k]) per block
//   af_finalize     one block: Rbar = mean R, RMS(U) = sqrt(Rbar sum / NK),
//                   RMS(W) = sqrt(sum c^2 / NK) / s_w, alpha, the clipped
//                   code-domain step and the weight decay, into 8 floats
//   af_apply        third read of G: v = R[n] C[k] / Rbar, u = g / sqrt(v),
//                   x = c decay - step u, then SR (Eq. 1) and the clamp (Eq. 5)
//
// Every reduction has a fixed shape and order, so results do not depend on
// scheduling.  Codes may be int8 or 2-bit packed ternary.
#include "dqt_internal.h"

namespace dqt {

namespace {

constexpr int kThreads = 256;
constexpr int kRowsPerSlab = 32;           // rows per af_sq/usq block
constexpr int kColsPerBlock = kThreads * 4;  // 1024 columns per block (float4 per thread)

__device__ __forceinline__ char4 load_codes4(const int8_t* W, bool packed, int64_t e) {
  return packed ? tern_unpack4(reinterpret_cast<const uint8_t*>(W)[e >> 2])
                : *reinterpret_cast<const char4*>(W + e);
}

template <typename T>
__device__ __forceinline__ T block_sum(T v, T* sh) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  T s = 0;
  if (threadIdx.x == 0)
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) s += sh[w];
  return s;  // valid in thread 0
}

__global__ void __launch_bounds__(kThreads)
    af_sq_partials_kernel(const float* __restrict__ G, const int8_t* __restrict__ W, bool packed,
                          int N, int K, float eps1, float* __restrict__ rowpart,
                          float* __restrict__ colpart, unsigned long long* __restrict__ cpart) {
  __shared__ unsigned long long sh[kThreads / 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k0 = blockIdx.x * kColsPerBlock + threadIdx.x * 4;
  const int n0 = blockIdx.y * kRowsPerSlab;
  const bool col_ok = k0 < K;  // K is a multiple of 4: the whole float4 is in range
  float cs[4] = {0.f, 0.f, 0.f, 0.f};
  unsigned long long csq = 0;
  const int chunk = blockIdx.x * (kColsPerBlock / 128) + warp;  // this warp's 128-column chunk
  const int nchunks = (K + 127) / 128;
  for (int r = 0; r < kRowsPerSlab; ++r) {
    const int n = n0 + r;
    if (n >= N) break;
    float rs = 0.f;
    if (col_ok) {
      const int64_t e = static_cast<int64_t>(n) * K + k0;
      const float4 g = __ldcs(reinterpret_cast<const float4*>(G + e));
      const float q0 = __fadd_rn(__fmul_rn(g.x, g.x), eps1);
      const float q1 = __fadd_rn(__fmul_rn(g.y, g.y), eps1);
      const float q2 = __fadd_rn(__fmul_rn(g.z, g.z), eps1);
      const float q3 = __fadd_rn(__fmul_rn(g.w, g.w), eps1);
      cs[0] += q0;
      cs[1] += q1;
      cs[2] += q2;
      cs[3] += q3;
      rs = (q0 + q1) + (q2 + q3);
      const char4 c = load_codes4(W, packed, e);
      csq += static_cast<unsigned long long>(c.x * c.x + c.y * c.y + c.z * c.z + c.w * c.w);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) rs += __shfl_xor_sync(0xffffffffu, rs, off);
    if (lane == 0 && chunk < nchunks) rowpart[static_cast<int64_t>(chunk) * N + n] = rs;
  }
  if (col_ok) {
    float* cp = colpart + static_cast<int64_t>(blockIdx.y) * K + k0;
    *reinterpret_cast<float4*>(cp) = make_float4(cs[0], cs[1], cs[2], cs[3]);
  }
  const unsigned long long tot = block_sum(csq, sh);
  if (threadIdx.x == 0) cpart[static_cast<int64_t>(blockIdx.y) * gridDim.x + blockIdx.x] = tot;
}

__global__ void __launch_bounds__(kThreads)
    af_moments_kernel(const float* __restrict__ rowpart, const float* __restrict__ colpart,
                      int nchunks, int nslabs, int N, int K, float b2, float omb2,
                      float* __restrict__ R, float* __restrict__ C) {
  const int t = blockIdx.x * kThreads + threadIdx.x;
  if (t < N) {
    float s = 0.f;
    for (int j = 0; j < nchunks; ++j) s += rowpart[static_cast<int64_t>(j) * N + t];
    const float mean = __fdiv_rn(s, static_cast<float>(K));
    R[t] = __fadd_rn(__fmul_rn(b2, R[t]), __fmul_rn(omb2, mean));
  } else if (t < N + K) {
    const int k = t - N;
    float s = 0.f;
    for (int j = 0; j < nslabs; ++j) s += colpart[static_cast<int64_t>(j) * K + k];
    const float mean = __fdiv_rn(s, static_cast<float>(N));
    C[k] = __fadd_rn(__fmul_rn(b2, C[k]), __fmul_rn(omb2, mean));
  }
}

__global__ void __launch_bounds__(kThreads)
    af_usq_partials_kernel(const float* __restrict__ G, const float* __restrict__ R,
                           const float* __restrict__ C, int N, int K, float* __restrict__ upart) {
  __shared__ float sh[kThreads / 32];
  const int k0 = blockIdx.x * kColsPerBlock + threadIdx.x * 4;
  const int n0 = blockIdx.y * kRowsPerSlab;
  float acc = 0.f;
  if (k0 < K) {
    const float4 c = *reinterpret_cast<const float4*>(C + k0);
    const float ic[4] = {__frcp_rn(c.x), __frcp_rn(c.y), __frcp_rn(c.z), __frcp_rn(c.w)};
    for (int r = 0; r < kRowsPerSlab; ++r) {
      const int n = n0 + r;
      if (n >= N) break;
      const float ir = __frcp_rn(R[n]);
      const float4 g = __ldcs(reinterpret_cast<const float4*>(G + static_cast<int64_t>(n) * K + k0));
      const float t = g.x * g.x * ic[0] + g.y * g.y * ic[1] + g.z * g.z * ic[2] + g.w * g.w * ic[3];
      acc += t * ir;
    }
  }
  const float tot = block_sum(acc, sh);
  if (threadIdx.x == 0) upart[static_cast<int64_t>(blockIdx.y) * gridDim.x + blockIdx.x] = tot;
}

// One block: the step's scalars.  out = {Rbar, step, decay, rms_u, rms_x, alpha}.
__global__ void __launch_bounds__(1024)
    af_finalize_kernel(const float* __restrict__ R, int N, int K, const float* __restrict__ upart,
                       const unsigned long long* __restrict__ cpart, int nparts, float s_w,
                       float rho, float eps2, float clip_d, int scale_parameter,
                       float weight_decay, float* __restrict__ out) {
  __shared__ double shd[32];
  __shared__ unsigned long long shu[32];
  double rs = 0.0, us = 0.0;
  unsigned long long cs = 0;
  for (int i = threadIdx.x; i < N; i += blockDim.x) rs += static_cast<double>(R[i]);
  for (int i = threadIdx.x; i < nparts; i += blockDim.x) {
    us += static_cast<double>(upart[i]);
    cs += cpart[i];
  }
  rs = block_sum(rs, shd);
  __syncthreads();
  us = block_sum(us, shd);
  __syncthreads();
  cs = block_sum(cs, shu);
  if (threadIdx.x == 0) {
    const double nk = static_cast<double>(N) * static_cast<double>(K);
    const double rbar = rs / static_cast<double>(N);
    const double rms_u = sqrt(rbar * us / nk);
    const double rms_x = sqrt(static_cast<double>(cs) / nk) / static_cast<double>(s_w);
    const double alpha =
        static_cast<double>(rho) * (scale_parameter ? fmax(static_cast<double>(eps2), rms_x) : 1.0);
    const double div = fmax(1.0, rms_u / static_cast<double>(clip_d));
    out[0] = static_cast<float>(rbar);
    out[1] = static_cast<float>(static_cast<double>(s_w) * alpha / div);
    out[2] = static_cast<float>(1.0 - static_cast<double>(weight_decay) * alpha);
    out[3] = static_cast<float>(rms_u);
    out[4] = static_cast<float>(rms_x);
    out[5] = static_cast<float>(alpha);
  }
}

struct ApplyArgs {
  int32_t qmin, qmax, round_mode;
  uint32_t step_lo, tensor_id, key0, key1;
};

__global__ void __launch_bounds__(kThreads)
    af_apply_kernel(const float* __restrict__ G, int8_t* __restrict__ W, bool packed,
                    const float* __restrict__ R, const float* __restrict__ C,
                    const float* __restrict__ scal, int N, int K, const ApplyArgs a,
                    unsigned long long* changed) {
  const float rbar = scal[0], step = scal[1], decay = scal[2];
  const int64_t ngroups = (static_cast<int64_t>(N) * K) >> 2;  // K % 4 == 0: no ragged group
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  uint8_t* Wp = reinterpret_cast<uint8_t*>(W);
  uint32_t n_changed = 0;
  for (int64_t gi = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; gi < ngroups;
       gi += stride) {
    const int64_t e = gi << 2;
    const int n = static_cast<int>(e / K);
    const int k = static_cast<int>(e - static_cast<int64_t>(n) * K);
    const float4 g = __ldcs(reinterpret_cast<const float4*>(G + e));
    const float4 c4 = *reinterpret_cast<const float4*>(C + k);
    const float rn = R[n];
    const char4 cc = load_codes4(W, packed, e);
    uint4 w = make_uint4(0, 0, 0, 0);
    if (a.round_mode == 0) w = sr_words(static_cast<uint64_t>(gi), a.step_lo, a.tensor_id, a.key0, a.key1);
    const float gs[4] = {g.x, g.y, g.z, g.w};
    const float cs[4] = {c4.x, c4.y, c4.z, c4.w};
    const int32_t c0[4] = {cc.x, cc.y, cc.z, cc.w};
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
    int32_t r[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float v = __fdiv_rn(__fmul_rn(rn, cs[j]), rbar);
      const float u = __fdiv_rn(gs[j], __fsqrt_rn(v));
      const float x = __fsub_rn(__fmul_rn(static_cast<float>(c0[j]), decay), __fmul_rn(step, u));
      r[j] = sr_round(x, ws[j], a.round_mode, a.qmin, a.qmax);
      n_changed += (r[j] != c0[j]);
    }
    if (packed)
      Wp[gi] = static_cast<uint8_t>(tern_pack4(r[0], r[1], r[2], r[3]));
    else
      *reinterpret_cast<char4*>(W + e) =
          make_char4(static_cast<signed char>(r[0]), static_cast<signed char>(r[1]),
                     static_cast<signed char>(r[2]), static_cast<signed char>(r[3]));
  }
  if (changed) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) n_changed += __shfl_xor_sync(0xffffffffu, n_changed, off);
    if ((threadIdx.x & 31) == 0 && n_changed)
      atomicAdd(changed, static_cast<unsigned long long>(n_changed));
  }
}

struct Layout {
  int nchunks, nslabs, gx, nparts;
  size_t row_off, col_off, cpart_off, upart_off, scal_off, bytes;
};

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

Layout layout(int64_t N, int64_t K) {
  Layout L{};
  L.nchunks = static_cast<int>((K + 127) / 128);
  L.nslabs = static_cast<int>((N + kRowsPerSlab - 1) / kRowsPerSlab);
  L.gx = static_cast<int>((K + kColsPerBlock - 1) / kColsPerBlock);
  L.nparts = L.gx * L.nslabs;
  L.row_off = 0;
  L.col_off = align256(L.row_off + static_cast<size_t>(L.nchunks) * N * 4);
  L.cpart_off = align256(L.col_off + static_cast<size_t>(L.nslabs) * K * 4);
  L.upart_off = align256(L.cpart_off + static_cast<size_t>(L.nparts) * 8);
  L.scal_off = align256(L.upart_off + static_cast<size_t>(L.nparts) * 4);
  L.bytes = align256(L.scal_off + 8 * 4);
  return L;
}

}  // namespace

size_t adafactor_stats_ws(int64_t N, int64_t K) { return layout(N, K).bytes; }
size_t adafactor_scalars_offset(int64_t N, int64_t K) { return layout(N, K).scal_off; }

int launch_adafactor_stats(const float* G, const int8_t* W, bool packed, float s_w, float* R,
                           float* C, const AdafactorConsts& h, int64_t N, int64_t K, void* ws,
                           float* scalars_out, cudaStream_t stream) {
  const Layout L = layout(N, K);
  uint8_t* base = static_cast<uint8_t*>(ws);
  float* rowpart = reinterpret_cast<float*>(base + L.row_off);
  float* colpart = reinterpret_cast<float*>(base + L.col_off);
  unsigned long long* cpart = reinterpret_cast<unsigned long long*>(base + L.cpart_off);
  float* upart = reinterpret_cast<float*>(base + L.upart_off);
  float* scal = scalars_out ? scalars_out : reinterpret_cast<float*>(base + L.scal_off);
  const int n = static_cast<int>(N), k = static_cast<int>(K);
  const dim3 grid(L.gx, L.nslabs);
  af_sq_partials_kernel<<<grid, kThreads, 0, stream>>>(G, W, packed, n, k, h.eps1, rowpart,
                                                       colpart, cpart);
  const int64_t nm = N + K;
  af_moments_kernel<<<static_cast<int>((nm + kThreads - 1) / kThreads), kThreads, 0, stream>>>(
      rowpart, colpart, L.nchunks, L.nslabs, n, k, h.b2, h.omb2, R, C);
  af_usq_partials_kernel<<<grid, kThreads, 0, stream>>>(G, R, C, n, k, upart);
  af_finalize_kernel<<<1, 1024, 0, stream>>>(R, n, k, upart, cpart, L.nparts, s_w, h.rho, h.eps2,
                                             h.clip_d, h.scale_parameter, h.weight_decay, scal);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_adafactor_apply(const float* G, int8_t* W, bool packed, const float* R, const float* C,
                           const float* scalars, const UpdateConsts& uc, int64_t N, int64_t K,
                           unsigned long long* changed, cudaStream_t stream) {
  ApplyArgs a;
  a.qmin = uc.qmin;
  a.qmax = uc.qmax;
  a.round_mode = uc.round_mode;
  a.step_lo = uc.step_lo;
  a.tensor_id = uc.tensor_id;
  a.key0 = uc.key0;
  a.key1 = uc.key1;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t groups = (N * K) >> 2;
  int64_t blocks = (groups + kThreads - 1) / kThreads;
  if (blocks > static_cast<int64_t>(sms) * 8) blocks = static_cast<int64_t>(sms) * 8;
  if (blocks < 1) blocks = 1;
  af_apply_kernel<<<static_cast<int>(blocks), kThreads, 0, stream>>>(
      G, W, packed, R, C, scalars, static_cast<int>(N), static_cast<int>(K), a, changed);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

}  // namespace dqt

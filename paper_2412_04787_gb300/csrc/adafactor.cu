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
//   af_factors      one block: Rbar = mean R, and the inverse square root of
//                   the rank-one estimate R C / Rbar as a row factor
//                   a[n] = 1 / sqrt(R[n] / Rbar) times a column factor
//                   b[k] = 1 / sqrt(C[k])
//   af_usq_partials second read of G: sum of u^2, u = (g a[n]) b[k], per block
//   af_finalize     one block: RMS(u), RMS(W) = sqrt(sum c^2 / NK) / s_w,
//                   alpha, the clipped code-domain step and the weight decay
//   af_apply        third read of G: u = (g a[n]) b[k], x = c decay - step u,
//                   then SR (Eq. 1) and the clamp (Eq. 5): two multiplies per
//                   weight besides the rounding, no division or square root
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

// Rows are taken kUnroll at a time: all their loads are issued before any is
// used, and their warp reductions interleave.  The codes are read only when
// the parameter RMS is needed (need_csq).
constexpr int kUnroll = 4;

__global__ void __launch_bounds__(kThreads, 4)
    af_sq_partials_kernel(const float* __restrict__ G, const int8_t* __restrict__ W, bool packed,
                          bool need_csq, int N, int K, float eps1, float* __restrict__ rowpart,
                          float* __restrict__ colpart, unsigned long long* __restrict__ cpart) {
  __shared__ unsigned long long sh[kThreads / 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k0 = blockIdx.x * kColsPerBlock + threadIdx.x * 4;
  const int n0 = blockIdx.y * kRowsPerSlab;
  const bool col_ok = k0 < K;  // K is a multiple of 4: the whole float4 is in range
  float cs[4] = {0.f, 0.f, 0.f, 0.f};
  uint32_t csq = 0;  // at most 32 rows x 4 codes x 128^2 per thread
  const int chunk = blockIdx.x * (kColsPerBlock / 128) + warp;  // this warp's 128-column chunk
  const int nchunks = (K + 127) / 128;
  for (int r0 = 0; r0 < kRowsPerSlab && n0 + r0 < N; r0 += kUnroll) {
    float4 g[kUnroll];
    char4 c[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int n = n0 + r0 + u;
      g[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      c[u] = make_char4(0, 0, 0, 0);
      if (col_ok && n < N) {
        const int64_t e = static_cast<int64_t>(n) * K + k0;
        g[u] = __ldcs(reinterpret_cast<const float4*>(G + e));
        if (need_csq) c[u] = load_codes4(W, packed, e);
      }
    }
    float rs[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      rs[u] = 0.f;
      if (col_ok && n0 + r0 + u < N) {
        const float q0 = __fadd_rn(__fmul_rn(g[u].x, g[u].x), eps1);
        const float q1 = __fadd_rn(__fmul_rn(g[u].y, g[u].y), eps1);
        const float q2 = __fadd_rn(__fmul_rn(g[u].z, g[u].z), eps1);
        const float q3 = __fadd_rn(__fmul_rn(g[u].w, g[u].w), eps1);
        cs[0] += q0;
        cs[1] += q1;
        cs[2] += q2;
        cs[3] += q3;
        rs[u] = (q0 + q1) + (q2 + q3);
        csq += static_cast<uint32_t>(c[u].x * c[u].x + c[u].y * c[u].y + c[u].z * c[u].z +
                                     c[u].w * c[u].w);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) rs[u] += __shfl_xor_sync(0xffffffffu, rs[u], off);
    if (lane == 0 && chunk < nchunks)
#pragma unroll
      for (int u = 0; u < kUnroll; ++u)
        if (n0 + r0 + u < N) rowpart[static_cast<int64_t>(chunk) * N + n0 + r0 + u] = rs[u];
  }
  if (col_ok) {
    float* cp = colpart + static_cast<int64_t>(blockIdx.y) * K + k0;
    *reinterpret_cast<float4*>(cp) = make_float4(cs[0], cs[1], cs[2], cs[3]);
  }
  const unsigned long long tot = block_sum(static_cast<unsigned long long>(csq), sh);
  if (threadIdx.x == 0) cpart[static_cast<int64_t>(blockIdx.y) * gridDim.x + blockIdx.x] = tot;
}

// The first row_blocks blocks finish the row means (one thread per row, its
// 128-column chunk partials in order); the others the column means: 32
// columns per block, eight threads per column each summing every eighth
// 32-row slab partial, then the eight sums combined in order in shared memory.
__global__ void __launch_bounds__(kThreads)
    af_moments_kernel(const float* __restrict__ rowpart, const float* __restrict__ colpart,
                      int nchunks, int nslabs, int N, int K, int row_blocks, float b2, float omb2,
                      float* __restrict__ R, float* __restrict__ C) {
  if (static_cast<int>(blockIdx.x) < row_blocks) {
    const int t = blockIdx.x * kThreads + threadIdx.x;
    if (t >= N) return;
    float s = 0.f;
    for (int j = 0; j < nchunks; ++j) s += rowpart[static_cast<int64_t>(j) * N + t];
    const float mean = __fdiv_rn(s, static_cast<float>(K));
    R[t] = __fadd_rn(__fmul_rn(b2, R[t]), __fmul_rn(omb2, mean));
    return;
  }
  __shared__ float part[8][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const int k = (blockIdx.x - row_blocks) * 32 + tx;
  float s0 = 0.f, s1 = 0.f;
  if (k < K) {
    int j = ty;
    for (; j + 8 < nslabs; j += 16) {  // two loads in flight per thread
      s0 += colpart[static_cast<int64_t>(j) * K + k];
      s1 += colpart[static_cast<int64_t>(j + 8) * K + k];
    }
    if (j < nslabs) s0 += colpart[static_cast<int64_t>(j) * K + k];
  }
  part[ty][tx] = s0 + s1;
  __syncthreads();
  if (ty == 0 && k < K) {
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) s += part[i][tx];
    const float mean = __fdiv_rn(s, static_cast<float>(N));
    C[k] = __fadd_rn(__fmul_rn(b2, C[k]), __fmul_rn(omb2, mean));
  }
}

// Rbar (fixed-order fp64 sum of R, rounded once to fp32; every block forms
// the same sum), then this block's slice of the factors a[n] = 1 / sqrt(R[n] /
// Rbar) and b[k] = 1 / sqrt(C[k]) over the concatenated index n, then N + k,
// each from correctly rounded fp32 operations.
__global__ void __launch_bounds__(kThreads)
    af_factors_kernel(const float* __restrict__ R, const float* __restrict__ C, int N, int K,
                      float* __restrict__ a, float* __restrict__ b, float* __restrict__ scal) {
  __shared__ double shd[kThreads / 32];
  __shared__ float rbar_s;
  double rs = 0.0;
  for (int i = threadIdx.x; i < N; i += kThreads) rs += static_cast<double>(R[i]);
  rs = block_sum(rs, shd);
  if (threadIdx.x == 0) {
    rbar_s = static_cast<float>(rs / static_cast<double>(N));
    if (blockIdx.x == 0) scal[0] = rbar_s;
  }
  __syncthreads();
  const float rbar = rbar_s;
  const int i = blockIdx.x * kThreads + threadIdx.x;
  if (i < N)
    a[i] = __fdiv_rn(1.0f, __fsqrt_rn(__fdiv_rn(R[i], rbar)));
  else if (i < N + K)
    b[i - N] = __fdiv_rn(1.0f, __fsqrt_rn(C[i - N]));
}

__device__ __forceinline__ float af_u(float g, float an, float bk) {
  return __fmul_rn(__fmul_rn(g, an), bk);
}

__global__ void __launch_bounds__(kThreads)
    af_usq_partials_kernel(const float* __restrict__ G, const float* __restrict__ a,
                           const float* __restrict__ b, int N, int K, float* __restrict__ upart) {
  __shared__ float sh[kThreads / 32];
  const int k0 = blockIdx.x * kColsPerBlock + threadIdx.x * 4;
  const int n0 = blockIdx.y * kRowsPerSlab;
  float acc = 0.f;
  if (k0 < K) {
    const float4 bk = *reinterpret_cast<const float4*>(b + k0);
    for (int r0 = 0; r0 < kRowsPerSlab && n0 + r0 < N; r0 += kUnroll) {
      float4 g[kUnroll];
      float an[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int n = n0 + r0 + u;
        g[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        an[u] = 0.f;
        if (n < N) {
          g[u] = __ldcs(reinterpret_cast<const float4*>(G + static_cast<int64_t>(n) * K + k0));
          an[u] = a[n];
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const float u0 = af_u(g[u].x, an[u], bk.x), u1 = af_u(g[u].y, an[u], bk.y);
        const float u2 = af_u(g[u].z, an[u], bk.z), u3 = af_u(g[u].w, an[u], bk.w);
        acc += (u0 * u0 + u1 * u1) + (u2 * u2 + u3 * u3);
      }
    }
  }
  const float tot = block_sum(acc, sh);
  if (threadIdx.x == 0) upart[static_cast<int64_t>(blockIdx.y) * gridDim.x + blockIdx.x] = tot;
}

// One block: the step's scalars.  out = {Rbar (already there), step, decay,
// rms_u, rms_x, alpha}.
__global__ void __launch_bounds__(kThreads)
    af_finalize_kernel(int N, int K, const float* __restrict__ upart,
                       const unsigned long long* __restrict__ cpart, int nparts, float s_w,
                       float rho, float eps2, float clip_d, int scale_parameter,
                       float weight_decay, float* __restrict__ out) {
  __shared__ double shd[kThreads / 32];
  __shared__ unsigned long long shu[kThreads / 32];
  double us = 0.0;
  unsigned long long cs = 0;
  for (int i = threadIdx.x; i < nparts; i += blockDim.x) {
    us += static_cast<double>(upart[i]);
    cs += cpart[i];
  }
  us = block_sum(us, shd);
  __syncthreads();
  cs = block_sum(cs, shu);
  if (threadIdx.x == 0) {
    const double nk = static_cast<double>(N) * static_cast<double>(K);
    const double rms_u = sqrt(us / nk);
    const double rms_x = sqrt(static_cast<double>(cs) / nk) / static_cast<double>(s_w);
    const double alpha =
        static_cast<double>(rho) * (scale_parameter ? fmax(static_cast<double>(eps2), rms_x) : 1.0);
    const double div = fmax(1.0, rms_u / static_cast<double>(clip_d));
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

template <bool WIDE>  // WIDE: N * K >= 2^32, 64-bit index arithmetic
__global__ void __launch_bounds__(kThreads)
    af_apply_kernel(const float* __restrict__ G, int8_t* __restrict__ W, bool packed,
                    const float* __restrict__ fa, const float* __restrict__ fb,
                    const float* __restrict__ scal, int N, int K, const ApplyArgs a,
                    unsigned long long* changed) {
  const float step = scal[1], decay = scal[2];
  const int64_t ngroups = (static_cast<int64_t>(N) * K) >> 2;  // K % 4 == 0: no ragged group
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  uint8_t* Wp = reinterpret_cast<uint8_t*>(W);
  uint32_t n_changed = 0;
  for (int64_t gi = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; gi < ngroups;
       gi += stride) {
    const int64_t e = gi << 2;
    int n, k;
    if (WIDE) {
      n = static_cast<int>(e / K);
      k = static_cast<int>(e - static_cast<int64_t>(n) * K);
    } else {
      const uint32_t e32 = static_cast<uint32_t>(e);
      n = static_cast<int>(e32 / static_cast<uint32_t>(K));
      k = static_cast<int>(e32 - static_cast<uint32_t>(n) * static_cast<uint32_t>(K));
    }
    const float4 g = __ldcs(reinterpret_cast<const float4*>(G + e));
    const float4 b4 = *reinterpret_cast<const float4*>(fb + k);
    const float an = fa[n];
    const char4 cc = load_codes4(W, packed, e);
    uint4 w = make_uint4(0, 0, 0, 0);
    if (a.round_mode == 0) w = sr_words(static_cast<uint64_t>(gi), a.step_lo, a.tensor_id, a.key0, a.key1);
    const float gs[4] = {g.x, g.y, g.z, g.w};
    const float bs[4] = {b4.x, b4.y, b4.z, b4.w};
    const int32_t c0[4] = {cc.x, cc.y, cc.z, cc.w};
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
    int32_t r[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float u = af_u(gs[j], an, bs[j]);
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
  size_t row_off, col_off, cpart_off, upart_off, scal_off, a_off, b_off, bytes;
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
  L.a_off = align256(L.scal_off + 8 * 4);
  L.b_off = align256(L.a_off + static_cast<size_t>(N) * 4);
  L.bytes = align256(L.b_off + static_cast<size_t>(K) * 4);
  return L;
}

}  // namespace

size_t adafactor_stats_ws(int64_t N, int64_t K) { return layout(N, K).bytes; }

AdafactorBufs adafactor_bufs(void* ws, int64_t N, int64_t K) {
  const Layout L = layout(N, K);
  uint8_t* base = static_cast<uint8_t*>(ws);
  AdafactorBufs b;
  b.a = reinterpret_cast<float*>(base + L.a_off);
  b.b = reinterpret_cast<float*>(base + L.b_off);
  b.scalars = reinterpret_cast<float*>(base + L.scal_off);
  return b;
}

int launch_adafactor_stats(const float* G, const int8_t* W, bool packed, float s_w, float* R,
                           float* C, const AdafactorConsts& h, int64_t N, int64_t K, void* ws,
                           float* a_out, float* b_out, float* scalars_out, cudaStream_t stream) {
  const Layout L = layout(N, K);
  uint8_t* base = static_cast<uint8_t*>(ws);
  float* rowpart = reinterpret_cast<float*>(base + L.row_off);
  float* colpart = reinterpret_cast<float*>(base + L.col_off);
  unsigned long long* cpart = reinterpret_cast<unsigned long long*>(base + L.cpart_off);
  float* upart = reinterpret_cast<float*>(base + L.upart_off);
  float* scal = scalars_out;
  const int n = static_cast<int>(N), k = static_cast<int>(K);
  const dim3 grid(L.gx, L.nslabs);
  af_sq_partials_kernel<<<grid, kThreads, 0, stream>>>(G, W, packed, h.scale_parameter != 0, n, k,
                                                       h.eps1, rowpart, colpart, cpart);
  const int row_blocks = (n + kThreads - 1) / kThreads;
  const int col_blocks = (k + 31) / 32;
  af_moments_kernel<<<row_blocks + col_blocks, kThreads, 0, stream>>>(
      rowpart, colpart, L.nchunks, L.nslabs, n, k, row_blocks, h.b2, h.omb2, R, C);
  af_factors_kernel<<<(n + k + kThreads - 1) / kThreads, kThreads, 0, stream>>>(R, C, n, k, a_out,
                                                                              b_out, scal);
  af_usq_partials_kernel<<<grid, kThreads, 0, stream>>>(G, a_out, b_out, n, k, upart);
  af_finalize_kernel<<<1, kThreads, 0, stream>>>(n, k, upart, cpart, L.nparts, s_w, h.rho, h.eps2,
                                             h.clip_d, h.scale_parameter, h.weight_decay, scal);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_adafactor_apply(const float* G, int8_t* W, bool packed, const float* fa,
                           const float* fb, const float* scalars, const UpdateConsts& uc,
                           int64_t N, int64_t K, unsigned long long* changed,
                           cudaStream_t stream) {
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
  if (N * K >= (int64_t(1) << 32))
    af_apply_kernel<true><<<static_cast<int>(blocks), kThreads, 0, stream>>>(
        G, W, packed, fa, fb, scalars, static_cast<int>(N), static_cast<int>(K), a, changed);
  else
    af_apply_kernel<false><<<static_cast<int>(blocks), kThreads, 0, stream>>>(
        G, W, packed, fa, fb, scalars, static_cast<int>(N), static_cast<int>(K), a, changed);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

}  // namespace dqt

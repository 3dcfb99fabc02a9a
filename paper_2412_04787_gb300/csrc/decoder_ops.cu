// Decoder support kernels (not part of the DQT method): the rotary position
// embedding and the token cross-entropy of the LLaMA-structured decoder built
// around the BitLinear layers, each one HBM-bound pass over bf16 data with
// fp32 arithmetic, in place of chains of PyTorch elementwise kernels with fp32
// intermediates in HBM.
//
//   rope_kernel      y = x rotated pairwise by the position angle (LLaMA:
//                    interleaved pairs (x[2i], x[2i+1]) as complex numbers
//                    times exp(i theta)), or by -theta for the backward
//   ce_fwd_kernel    per row: lse = log sum_v exp(x_v), loss = lse - x_target
//   ce_bwd_kernel    dx_v = (exp(x_v - lse) - [v == target]) * scale
//   swiglu_kernel    h = silu(g) u, and its backward dg, du
//   rmsnorm_*        y = x rstd w with rstd = 1 / sqrt(mean(x^2) + eps) per
//                    row, and its backward (dx per row; dw as per-warp partial
//                    sums reduced in a fixed order)
#include <cuda_bf16.h>

#include "dqt_internal.h"

namespace dqt {

namespace {

constexpr int kRopeThreads = 256;
constexpr int kCeThreads = 256;

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// One 16-byte vector (four pairs of one head) per thread step.  cs holds
// (cos, sin) per position and pair: fp32 [S, D/2, 2].
template <bool INV>
__global__ void __launch_bounds__(kRopeThreads)
    rope_kernel(const uint4* __restrict__ x, uint4* __restrict__ y, const float4* __restrict__ cs,
                int64_t nvec, int64_t row_vecs, int64_t S, int64_t head_vecs) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kRopeThreads;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kRopeThreads + threadIdx.x; i < nvec;
       i += stride) {
    const int64_t row = i / row_vecs;
    const int64_t dv = (i - row * row_vecs) % head_vecs;  // vector within the head
    const int64_t pos = row % S;
    // four pairs = eight floats = two float4 of the table
    const float4* t = cs + (pos * head_vecs + dv) * 2;
    const float4 c01 = __ldg(t), c23 = __ldg(t + 1);
    const float cth[4] = {c01.x, c01.z, c23.x, c23.z};
    const float sth[4] = {INV ? -c01.y : c01.y, INV ? -c01.w : c01.w, INV ? -c23.y : c23.y,
                          INV ? -c23.w : c23.w};
    const uint4 v = x[i];
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float xe = bf16_lo(w[j]), xo = bf16_hi(w[j]);
      const float ye = __fsub_rn(__fmul_rn(xe, cth[j]), __fmul_rn(xo, sth[j]));
      const float yo = __fadd_rn(__fmul_rn(xe, sth[j]), __fmul_rn(xo, cth[j]));
      o[j] = pack_bf16x2(ye, yo);
    }
    y[i] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// (max, sum of exp(x - max)) pairs combine associatively
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  if (m2 > m) {
    s = s * expf(m - m2) + s2;
    m = m2;
  } else if (m2 != -INFINITY) {
    s += s2 * expf(m2 - m);
  }
}

__device__ __forceinline__ void lse_block(float& m, float& s, float* sh_m, float* sh_s) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1)
    lse_merge(m, s, __shfl_xor_sync(0xffffffffu, m, off), __shfl_xor_sync(0xffffffffu, s, off));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    sh_m[warp] = m;
    sh_s[warp] = s;
  }
  __syncthreads();
  if (warp == 0) {
    m = lane < kCeThreads / 32 ? sh_m[lane] : -INFINITY;
    s = lane < kCeThreads / 32 ? sh_s[lane] : 0.0f;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
      lse_merge(m, s, __shfl_xor_sync(0xffffffffu, m, off), __shfl_xor_sync(0xffffffffu, s, off));
  }
}

// One block per row; V a multiple of 8 (16-byte vectors of bf16).
__global__ void __launch_bounds__(kCeThreads)
    ce_fwd_kernel(const uint4* __restrict__ logits, const int64_t* __restrict__ tgt, int64_t V,
                  float* __restrict__ lse, float* __restrict__ row_loss) {
  __shared__ float sh_m[kCeThreads / 32], sh_s[kCeThreads / 32];
  const int64_t r = blockIdx.x;
  const int64_t nv = V >> 3;
  const uint4* row = logits + r * nv;
  float m = -INFINITY, s = 0.0f;
  // two vectors in flight per thread step
  for (int64_t i = threadIdx.x; i < nv; i += 2 * kCeThreads) {
    const bool two = i + kCeThreads < nv;
    const uint4 va = __ldcs(row + i);
    const uint4 vb = two ? __ldcs(row + i + kCeThreads) : va;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      if (h == 1 && !two) break;
      const uint4 v = h ? vb : va;
      const float f[8] = {bf16_lo(v.x), bf16_hi(v.x), bf16_lo(v.y), bf16_hi(v.y),
                          bf16_lo(v.z), bf16_hi(v.z), bf16_lo(v.w), bf16_hi(v.w)};
      float mv = f[0];
#pragma unroll
      for (int j = 1; j < 8; ++j) mv = fmaxf(mv, f[j]);
      float sv = 0.0f;
#pragma unroll
      for (int j = 0; j < 8; ++j) sv += expf(f[j] - mv);
      lse_merge(m, s, mv, sv);
    }
  }
  lse_block(m, s, sh_m, sh_s);
  if (threadIdx.x == 0) {
    const float l = m + logf(s);
    const int64_t t = tgt[r];
    const bool ok = t >= 0 && t < V;
    const uint16_t xt = ok ? reinterpret_cast<const uint16_t*>(row)[t] : 0;
    lse[r] = l;
    row_loss[r] = ok ? l - __uint_as_float(static_cast<uint32_t>(xt) << 16) : 0.0f;
  }
}

// One block per row; a row whose target is outside [0, V) gets zeros.
__global__ void __launch_bounds__(kCeThreads)
    ce_bwd_kernel(const uint4* __restrict__ logits, const int64_t* __restrict__ tgt,
                  const float* __restrict__ lse, const float* __restrict__ scale, int64_t V,
                  uint4* __restrict__ dlogits) {
  const int64_t r = blockIdx.x;
  const int64_t nv = V >> 3;
  const int64_t t = tgt[r];
  const bool ok = t >= 0 && t < V;
  const float l = lse[r];
  const float g = ok ? scale[0] : 0.0f;
  const uint4* row = logits + r * nv;
  uint4* drow = dlogits + r * nv;
  // two vectors in flight per thread step
  for (int64_t i0 = threadIdx.x; i0 < nv; i0 += 2 * kCeThreads) {
    const bool two = i0 + kCeThreads < nv;
    const uint4 va = __ldcs(row + i0);
    const uint4 vb = two ? __ldcs(row + i0 + kCeThreads) : va;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      if (h == 1 && !two) break;
      const int64_t i = i0 + h * kCeThreads;
      const uint4 v = h ? vb : va;
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
      uint32_t o[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t c = i * 8 + 2 * j;
        const float p0 = expf(bf16_lo(w[j]) - l) - (c == t ? 1.0f : 0.0f);
        const float p1 = expf(bf16_hi(w[j]) - l) - (c + 1 == t ? 1.0f : 0.0f);
        o[j] = pack_bf16x2(p0 * g, p1 * g);
      }
      __stcs(drow + i, make_uint4(o[0], o[1], o[2], o[3]));
    }
  }
}

constexpr int kEwThreads = 256;

// SwiGLU gate: h = g sigmoid(g) u in fp32 per element, one rounding to bf16;
// 8 elements (one 16-byte vector of each operand) per thread step.
__global__ void __launch_bounds__(kEwThreads)
    swiglu_kernel(const uint4* __restrict__ g, const uint4* __restrict__ u, uint4* __restrict__ h,
                  int64_t nvec) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kEwThreads;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kEwThreads + threadIdx.x; i < nvec;
       i += stride) {
    const uint4 gv = __ldcs(g + i), uv = __ldcs(u + i);
    const uint32_t gw[4] = {gv.x, gv.y, gv.z, gv.w}, uw[4] = {uv.x, uv.y, uv.z, uv.w};
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float g0 = bf16_lo(gw[j]), g1 = bf16_hi(gw[j]);
      const float s0 = 1.0f / (1.0f + expf(-g0)), s1 = 1.0f / (1.0f + expf(-g1));
      o[j] = pack_bf16x2(g0 * s0 * bf16_lo(uw[j]), g1 * s1 * bf16_hi(uw[j]));
    }
    h[i] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// Its backward: with s = sigmoid(g),
//   dg = dh u s (1 + g (1 - s)),   du = dh g s
__global__ void __launch_bounds__(kEwThreads)
    swiglu_bwd_kernel(const uint4* __restrict__ g, const uint4* __restrict__ u,
                      const uint4* __restrict__ dh, uint4* __restrict__ dg,
                      uint4* __restrict__ du, int64_t nvec) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kEwThreads;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kEwThreads + threadIdx.x; i < nvec;
       i += stride) {
    const uint4 gv = __ldcs(g + i), uv = __ldcs(u + i), hv = __ldcs(dh + i);
    const uint32_t gw[4] = {gv.x, gv.y, gv.z, gv.w}, uw[4] = {uv.x, uv.y, uv.z, uv.w},
                   hw[4] = {hv.x, hv.y, hv.z, hv.w};
    uint32_t og[4], ou[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      float rg[2], ru[2];
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const float gg = k ? bf16_hi(gw[j]) : bf16_lo(gw[j]);
        const float uu = k ? bf16_hi(uw[j]) : bf16_lo(uw[j]);
        const float d = k ? bf16_hi(hw[j]) : bf16_lo(hw[j]);
        const float s = 1.0f / (1.0f + expf(-gg));
        rg[k] = d * uu * s * (1.0f + gg * (1.0f - s));
        ru[k] = d * gg * s;
      }
      og[j] = pack_bf16x2(rg[0], rg[1]);
      ou[j] = pack_bf16x2(ru[0], ru[1]);
    }
    __stcs(dg + i, make_uint4(og[0], og[1], og[2], og[3]));
    __stcs(du + i, make_uint4(ou[0], ou[1], ou[2], ou[3]));
  }
}

constexpr int kNormWarps = 8;  // rows per block, one warp per row

// One warp per row; the row's D / 8 vectors are spread over the lanes,
// VPL = ceil(D / 256) vectors per lane held in registers.
template <int VPL>
__global__ void __launch_bounds__(32 * kNormWarps)
    rmsnorm_fwd_kernel(const uint4* __restrict__ x, const uint4* __restrict__ w, float eps,
                       int64_t rows, int nv, uint4* __restrict__ y, float* __restrict__ rstd) {
  const int lane = threadIdx.x & 31;
  const int64_t row = static_cast<int64_t>(blockIdx.x) * kNormWarps + (threadIdx.x >> 5);
  if (row >= rows) return;
  const uint4* xr = x + row * nv;
  uint4 xv[VPL];
  float ss = 0.0f;
#pragma unroll
  for (int k = 0; k < VPL; ++k) {
    const int c = lane + 32 * k;
    xv[k] = c < nv ? __ldcs(xr + c) : make_uint4(0, 0, 0, 0);
    const uint32_t a[4] = {xv[k].x, xv[k].y, xv[k].z, xv[k].w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float lo = bf16_lo(a[j]), hi = bf16_hi(a[j]);
      ss += lo * lo + hi * hi;
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
  const float r = 1.0f / sqrtf(ss / static_cast<float>(nv * 8) + eps);
  if (lane == 0) rstd[row] = r;
  uint4* yr = y + row * nv;
#pragma unroll
  for (int k = 0; k < VPL; ++k) {
    const int c = lane + 32 * k;
    if (c >= nv) break;
    const uint4 wv = __ldg(w + c);
    const uint32_t a[4] = {xv[k].x, xv[k].y, xv[k].z, xv[k].w};
    const uint32_t b[4] = {wv.x, wv.y, wv.z, wv.w};
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
      o[j] = pack_bf16x2(bf16_lo(a[j]) * r * bf16_lo(b[j]), bf16_hi(a[j]) * r * bf16_hi(b[j]));
    yr[c] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// Backward of y = x r w, r = rstd:
//   dx_j = r w_j dy_j - x_j r^3 (1/D) sum_k w_k dy_k x_k
//   dw_j = sum over rows of dy_j x_j r
// Each warp walks rows warp_id, warp_id + nwarps, ... and keeps its dw
// partial sums in registers; they go to part[warp_id, :] (fp32) at the end.
template <int VPL>
__global__ void __launch_bounds__(32 * kNormWarps)
    rmsnorm_bwd_kernel(const uint4* __restrict__ x, const uint4* __restrict__ w,
                       const float* __restrict__ rstd, const uint4* __restrict__ dy, int64_t rows,
                       int nv, uint4* __restrict__ dx, float* __restrict__ part) {
  const int lane = threadIdx.x & 31;
  const int64_t wid = static_cast<int64_t>(blockIdx.x) * kNormWarps + (threadIdx.x >> 5);
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kNormWarps;
  const float inv_d = 1.0f / static_cast<float>(nv * 8);
  // the gain vector is re-read per row from L1 (it is D * 2 bytes) rather
  // than held in registers next to the partial sums
  float acc[VPL][8];
#pragma unroll
  for (int k = 0; k < VPL; ++k)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[k][j] = 0.0f;
  for (int64_t row = wid; row < rows; row += nwarps) {
    const float r = rstd[row];
    uint4 xv[VPL], gv[VPL];
    float dot = 0.0f;
#pragma unroll
    for (int k = 0; k < VPL; ++k) {
      const int c = lane + 32 * k;
      xv[k] = c < nv ? __ldcs(x + row * nv + c) : make_uint4(0, 0, 0, 0);
      gv[k] = c < nv ? __ldcs(dy + row * nv + c) : make_uint4(0, 0, 0, 0);
      const uint4 wv = c < nv ? __ldg(w + c) : make_uint4(0, 0, 0, 0);
      const uint32_t a[4] = {xv[k].x, xv[k].y, xv[k].z, xv[k].w};
      const uint32_t g[4] = {gv[k].x, gv[k].y, gv[k].z, gv[k].w};
      const uint32_t b[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        dot += bf16_lo(b[j]) * bf16_lo(g[j]) * bf16_lo(a[j]);
        dot += bf16_hi(b[j]) * bf16_hi(g[j]) * bf16_hi(a[j]);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
    const float coef = r * r * r * dot * inv_d;
#pragma unroll
    for (int k = 0; k < VPL; ++k) {
      const int c = lane + 32 * k;
      if (c >= nv) break;
      const uint4 wv = __ldg(w + c);
      const uint32_t a[4] = {xv[k].x, xv[k].y, xv[k].z, xv[k].w};
      const uint32_t g[4] = {gv[k].x, gv[k].y, gv[k].z, gv[k].w};
      const uint32_t b[4] = {wv.x, wv.y, wv.z, wv.w};
      uint32_t o[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float x0 = bf16_lo(a[j]), x1 = bf16_hi(a[j]);
        const float g0 = bf16_lo(g[j]), g1 = bf16_hi(g[j]);
        o[j] = pack_bf16x2(r * bf16_lo(b[j]) * g0 - x0 * coef, r * bf16_hi(b[j]) * g1 - x1 * coef);
        acc[k][2 * j] += g0 * x0 * r;
        acc[k][2 * j + 1] += g1 * x1 * r;
      }
      __stcs(dx + row * nv + c, make_uint4(o[0], o[1], o[2], o[3]));
    }
  }
  float* pr = part + wid * static_cast<int64_t>(nv) * 8;
#pragma unroll
  for (int k = 0; k < VPL; ++k) {
    const int c = lane + 32 * k;
    if (c >= nv) break;
    float4* d = reinterpret_cast<float4*>(pr + c * 8);
    d[0] = make_float4(acc[k][0], acc[k][1], acc[k][2], acc[k][3]);
    d[1] = make_float4(acc[k][4], acc[k][5], acc[k][6], acc[k][7]);
  }
}

// dw_j = the sum of the P partial rows, rounded once to bf16, in a fixed
// order: a block covers 32 columns, warp k sums the partial rows p = k mod 8
// in increasing p, and the block adds the 8 warp sums in warp order.
__global__ void __launch_bounds__(256)
    rmsnorm_dw_kernel(const float* __restrict__ part, int64_t P, int D, uint16_t* __restrict__ dw) {
  __shared__ float sh[8][33];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int col = blockIdx.x * 32 + lane;
  float s = 0.0f;
  if (col < D)
    for (int64_t p = warp; p < P; p += 8) s += part[p * D + col];
  sh[warp][lane] = s;
  __syncthreads();
  if (warp == 0 && col < D) {
    float t = 0.0f;
#pragma unroll
    for (int k = 0; k < 8; ++k) t += sh[k][lane];
    const __nv_bfloat16 h = __float2bfloat16_rn(t);
    dw[col] = *reinterpret_cast<const uint16_t*>(&h);
  }
}

int norm_blocks_bwd() {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms;  // one block (8 warps) per SM: the partial sums take many registers
}

int grid_cap(int64_t items, int threads) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t b = (items + threads - 1) / threads;
  const int64_t cap = static_cast<int64_t>(sms) * 8;
  if (b > cap) b = cap;
  return static_cast<int>(b < 1 ? 1 : b);
}

}  // namespace

int launch_rope(const uint16_t* x, uint16_t* y, const float* cos_sin, int64_t rows, int64_t S,
                int64_t H, int64_t D, bool inverse, cudaStream_t stream) {
  const int64_t row_vecs = H * D / 8, head_vecs = D / 8;
  const int64_t nvec = rows * row_vecs;
  const int blocks = grid_cap(nvec, kRopeThreads);
  auto* xv = reinterpret_cast<const uint4*>(x);
  auto* yv = reinterpret_cast<uint4*>(y);
  auto* cv = reinterpret_cast<const float4*>(cos_sin);
  if (inverse)
    rope_kernel<true><<<blocks, kRopeThreads, 0, stream>>>(xv, yv, cv, nvec, row_vecs, S, head_vecs);
  else
    rope_kernel<false><<<blocks, kRopeThreads, 0, stream>>>(xv, yv, cv, nvec, row_vecs, S, head_vecs);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_ce_fwd(const uint16_t* logits, const int64_t* targets, int64_t M, int64_t V,
                  float* lse, float* row_loss, cudaStream_t stream) {
  ce_fwd_kernel<<<static_cast<unsigned>(M), kCeThreads, 0, stream>>>(
      reinterpret_cast<const uint4*>(logits), targets, V, lse, row_loss);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_ce_bwd(const uint16_t* logits, const int64_t* targets, const float* lse,
                  const float* scale, int64_t M, int64_t V, uint16_t* dlogits,
                  cudaStream_t stream) {
  ce_bwd_kernel<<<static_cast<unsigned>(M), kCeThreads, 0, stream>>>(
      reinterpret_cast<const uint4*>(logits), targets, lse, scale, V,
      reinterpret_cast<uint4*>(dlogits));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_swiglu(const uint16_t* g, const uint16_t* u, uint16_t* h, int64_t n,
                  cudaStream_t stream) {
  const int64_t nvec = n / 8;
  swiglu_kernel<<<grid_cap(nvec, kEwThreads), kEwThreads, 0, stream>>>(
      reinterpret_cast<const uint4*>(g), reinterpret_cast<const uint4*>(u),
      reinterpret_cast<uint4*>(h), nvec);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_swiglu_bwd(const uint16_t* g, const uint16_t* u, const uint16_t* dh, uint16_t* dg,
                      uint16_t* du, int64_t n, cudaStream_t stream) {
  const int64_t nvec = n / 8;
  swiglu_bwd_kernel<<<grid_cap(nvec, kEwThreads), kEwThreads, 0, stream>>>(
      reinterpret_cast<const uint4*>(g), reinterpret_cast<const uint4*>(u),
      reinterpret_cast<const uint4*>(dh), reinterpret_cast<uint4*>(dg),
      reinterpret_cast<uint4*>(du), nvec);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

size_t rmsnorm_bwd_ws(int64_t rows, int64_t D) {
  const int64_t blocks = norm_blocks_bwd();
  const int64_t need = (rows + kNormWarps - 1) / kNormWarps;
  const int64_t b = blocks < need ? blocks : need;
  return static_cast<size_t>(b * kNormWarps * D) * sizeof(float);
}

template <int VPL>
static int rms_launch(const uint16_t* x, const uint16_t* w, float eps, int64_t rows, int64_t D,
                      uint16_t* y, float* rstd, cudaStream_t stream) {
  const int nv = static_cast<int>(D / 8);
  const unsigned blocks = static_cast<unsigned>((rows + kNormWarps - 1) / kNormWarps);
  rmsnorm_fwd_kernel<VPL><<<blocks, 32 * kNormWarps, 0, stream>>>(
      reinterpret_cast<const uint4*>(x), reinterpret_cast<const uint4*>(w), eps, rows, nv,
      reinterpret_cast<uint4*>(y), rstd);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

template <int VPL>
static int rms_bwd_launch(const uint16_t* x, const uint16_t* w, const float* rstd,
                          const uint16_t* dy, int64_t rows, int64_t D, uint16_t* dx,
                          uint16_t* dw, float* part, cudaStream_t stream) {
  const int nv = static_cast<int>(D / 8);
  const int64_t need = (rows + kNormWarps - 1) / kNormWarps;
  const int64_t sms = norm_blocks_bwd();
  const unsigned blocks = static_cast<unsigned>(sms < need ? sms : need);
  rmsnorm_bwd_kernel<VPL><<<blocks, 32 * kNormWarps, 0, stream>>>(
      reinterpret_cast<const uint4*>(x), reinterpret_cast<const uint4*>(w), rstd,
      reinterpret_cast<const uint4*>(dy), rows, nv, reinterpret_cast<uint4*>(dx), part);
  const int64_t P = static_cast<int64_t>(blocks) * kNormWarps;
  rmsnorm_dw_kernel<<<static_cast<unsigned>((D + 31) / 32), 256, 0, stream>>>(
      part, P, static_cast<int>(D), dw);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_rmsnorm(const uint16_t* x, const uint16_t* w, float eps, int64_t rows, int64_t D,
                   uint16_t* y, float* rstd, cudaStream_t stream) {
  switch ((D / 8 + 31) / 32) {
    case 1: return rms_launch<1>(x, w, eps, rows, D, y, rstd, stream);
    case 2: return rms_launch<2>(x, w, eps, rows, D, y, rstd, stream);
    case 3: return rms_launch<3>(x, w, eps, rows, D, y, rstd, stream);
    case 4: return rms_launch<4>(x, w, eps, rows, D, y, rstd, stream);
    case 5: case 6: return rms_launch<6>(x, w, eps, rows, D, y, rstd, stream);
    case 7: case 8: return rms_launch<8>(x, w, eps, rows, D, y, rstd, stream);
    default: return 1;
  }
}

int launch_rmsnorm_bwd(const uint16_t* x, const uint16_t* w, const float* rstd,
                       const uint16_t* dy, int64_t rows, int64_t D, uint16_t* dx, uint16_t* dw,
                       float* part, cudaStream_t stream) {
  switch ((D / 8 + 31) / 32) {
    case 1: return rms_bwd_launch<1>(x, w, rstd, dy, rows, D, dx, dw, part, stream);
    case 2: return rms_bwd_launch<2>(x, w, rstd, dy, rows, D, dx, dw, part, stream);
    case 3: return rms_bwd_launch<3>(x, w, rstd, dy, rows, D, dx, dw, part, stream);
    case 4: return rms_bwd_launch<4>(x, w, rstd, dy, rows, D, dx, dw, part, stream);
    case 5: case 6: return rms_bwd_launch<6>(x, w, rstd, dy, rows, D, dx, dw, part, stream);
    case 7: case 8: return rms_bwd_launch<8>(x, w, rstd, dy, rows, D, dx, dw, part, stream);
    default: return 1;
  }
}

}  // namespace dqt

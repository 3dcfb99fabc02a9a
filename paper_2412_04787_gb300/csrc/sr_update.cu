// Standalone DQT weight update (Sec. 4.1 AdamW, Eq. 1 stochastic rounding,
// Eq. 5 W_hat = SR(W')) for a gradient already in memory: a streaming,
// HBM-bound kernel moving 22 bytes per weight (read g, m, v, c; write m, v, c).
//
// Each thread step handles one group of four consecutive weights, which is
// exactly one Philox4x32-10 block (element e uses word e % 4 of block e / 4),
// with 16-byte loads and stores of g, m, v and a 4-byte access to the codes
// (one byte when the codes are 2-bit packed ternary: a group is one byte).
#include <cuda_fp8.h>

#include "dqt_internal.h"

namespace dqt {

namespace {

constexpr int kThreads = 256;

// The gradient of element e is grad[e], or, with nsplit > 1 partial slabs of
// `slab` elements each (a split-T weight gradient), their sum taken in slab
// order; g_out (optional) receives that gradient.
__device__ __forceinline__ float4 slab_grad4(const float* __restrict__ grad, int nsplit,
                                             long long slab, int64_t e) {
  float4 g4 = __ldcs(reinterpret_cast<const float4*>(grad + e));
  for (int s = 1; s < nsplit; ++s) {
    const float4 h = __ldcs(reinterpret_cast<const float4*>(grad + s * slab + e));
    g4.x = __fadd_rn(g4.x, h.x);
    g4.y = __fadd_rn(g4.y, h.y);
    g4.z = __fadd_rn(g4.z, h.z);
    g4.w = __fadd_rn(g4.w, h.w);
  }
  return g4;
}

__device__ __forceinline__ float slab_grad1(const float* __restrict__ grad, int nsplit,
                                            long long slab, int64_t e) {
  float g = grad[e];
  for (int s = 1; s < nsplit; ++s) g = __fadd_rn(g, grad[s * slab + e]);
  return g;
}

__device__ __forceinline__ uint32_t e4m3x4(int32_t a, int32_t b, int32_t c, int32_t d) {
  const uint32_t lo = __nv_cvt_float2_to_fp8x2(
      make_float2(static_cast<float>(a), static_cast<float>(b)), __NV_SATFINITE, __NV_E4M3);
  const uint32_t hi = __nv_cvt_float2_to_fp8x2(
      make_float2(static_cast<float>(c), static_cast<float>(d)), __NV_SATFINITE, __NV_E4M3);
  return (lo & 0xFFFFu) | ((hi & 0xFFFFu) << 16);
}

// The E4M3 image of four new codes at element e: direct (img8_k == 0), or
// split into rows of img8_k codes, each row 2 img8_k bytes with 16 (c >> 4)
// at the code's column and c & 15 img8_k bytes later (e % 4 == 0 and img8_k
// % 4 == 0, so the four codes share a row).
__device__ __forceinline__ void store_e4m3_4(uint8_t* img8, int64_t img8_k, int64_t e, int32_t a,
                                             int32_t b, int32_t c, int32_t d) {
  if (!img8_k) {
    __stcs(reinterpret_cast<uint32_t*>(img8 + e), e4m3x4(a, b, c, d));
    return;
  }
  const int64_t h = e + (e / img8_k) * img8_k;
  __stcs(reinterpret_cast<uint32_t*>(img8 + h),
         e4m3x4(16 * (a >> 4), 16 * (b >> 4), 16 * (c >> 4), 16 * (d >> 4)));
  __stcs(reinterpret_cast<uint32_t*>(img8 + h + img8_k), e4m3x4(a & 15, b & 15, c & 15, d & 15));
}

// The bf16 and E4M3 images of four new codes (either pointer may be NULL).
__device__ __forceinline__ void store_images4(uint16_t* img, uint8_t* img8, int64_t img8_k,
                                              int64_t e, int32_t a, int32_t b, int32_t c,
                                              int32_t d) {
  if (img) {
    const __nv_bfloat162 lo = __floats2bfloat162_rn(static_cast<float>(a), static_cast<float>(b));
    const __nv_bfloat162 hi = __floats2bfloat162_rn(static_cast<float>(c), static_cast<float>(d));
    __stcs(reinterpret_cast<uint2*>(img + e),
           make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi)));
  }
  if (img8) store_e4m3_4(img8, img8_k, e, a, b, c, d);
}

// DEV: the constants are read from device memory (else the kernel's
// parameter space); SLABS: the gradient may be split into slabs and the
// summed gradient written out, and the images of the new codes (img bf16,
// img8 E4M3, direct or split as in store_e4m3_4; int8 codes only) written
// beside them.  The plain instance is the leanest stream.
template <bool packed, bool DEV, bool SLABS>
__global__ void __launch_bounds__(kThreads)
    sr_update_kernel(const float* __restrict__ grad, int nsplit, long long slab,
                     float* __restrict__ g_out, int8_t* __restrict__ W, float* __restrict__ m,
                     float* __restrict__ v, int64_t numel, const UpdateConsts uc_arg,
                     const UpdateConsts* __restrict__ uc_dev, unsigned long long* changed,
                     uint16_t* __restrict__ img, uint8_t* __restrict__ img8, int64_t img8_k) {
  uint8_t* Wp = reinterpret_cast<uint8_t*>(W);
  const UpdateConsts uc = DEV ? *uc_dev : uc_arg;
  const int64_t ngroups = numel >> 2;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  uint32_t n_changed = 0;
  for (int64_t gi = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; gi < ngroups;
       gi += stride) {
    const int64_t e = gi << 2;
    const float4 g4 = SLABS ? slab_grad4(grad, nsplit, slab, e)
                            : __ldcs(reinterpret_cast<const float4*>(grad + e));
    if (SLABS && g_out) __stcs(reinterpret_cast<float4*>(g_out + e), g4);
    float4 m4 = __ldcs(reinterpret_cast<const float4*>(m + e));
    float4 v4 = __ldcs(reinterpret_cast<const float4*>(v + e));
    const char4 c4 = packed ? tern_unpack4(Wp[gi]) : *reinterpret_cast<const char4*>(W + e);
    uint4 w = make_uint4(0, 0, 0, 0);
    if (uc.round_mode == 0)
      w = sr_words(global_blk(uc, static_cast<uint64_t>(gi)), uc.step_lo, uc.tensor_id, uc.key0,
                   uc.key1);
    const int32_t a = dqt_update_elem(uc, g4.x, c4.x, m4.x, v4.x, w.x);
    const int32_t b = dqt_update_elem(uc, g4.y, c4.y, m4.y, v4.y, w.y);
    const int32_t c = dqt_update_elem(uc, g4.z, c4.z, m4.z, v4.z, w.z);
    const int32_t d = dqt_update_elem(uc, g4.w, c4.w, m4.w, v4.w, w.w);
    n_changed += (a != c4.x) + (b != c4.y) + (c != c4.z) + (d != c4.w);
    if (packed)
      Wp[gi] = static_cast<uint8_t>(tern_pack4(a, b, c, d));
    else
      *reinterpret_cast<char4*>(W + e) =
          make_char4(static_cast<signed char>(a), static_cast<signed char>(b),
                     static_cast<signed char>(c), static_cast<signed char>(d));
    if (SLABS && !packed) store_images4(img, img8, img8_k, e, a, b, c, d);
    __stcs(reinterpret_cast<float4*>(m + e), m4);
    __stcs(reinterpret_cast<float4*>(v + e), v4);
  }
  // ragged tail: the last numel % 4 elements, one thread, scalar accesses
  if (blockIdx.x == 0 && threadIdx.x == 0 && (numel & 3)) {
    const int64_t gi = ngroups;
    uint4 w = make_uint4(0, 0, 0, 0);
    if (uc.round_mode == 0)
      w = sr_words(global_blk(uc, static_cast<uint64_t>(gi)), uc.step_lo, uc.tensor_id, uc.key0,
                   uc.key1);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
    const char4 pc = packed ? tern_unpack4(Wp[gi]) : make_char4(0, 0, 0, 0);
    int32_t pr[4] = {0, 0, 0, 0};  // packed: the unused fields of the last byte stay 0
    for (int64_t e = gi << 2; e < numel; ++e) {
      float mm = m[e], vv = v[e];
      const int j = static_cast<int>(e & 3);
      const int32_t c0 = packed ? (j == 0 ? pc.x : j == 1 ? pc.y : pc.z) : W[e];
      const float g = SLABS ? slab_grad1(grad, nsplit, slab, e) : grad[e];
      if (SLABS && g_out) g_out[e] = g;
      const int32_t r = dqt_update_elem(uc, g, c0, mm, vv, ws[j]);
      n_changed += (r != c0);
      if (packed) pr[j] = r;
      else W[e] = static_cast<int8_t>(r);
      if (SLABS && !packed && img) img[e] = __bfloat16_as_ushort(__float2bfloat16_rn(static_cast<float>(r)));
      if (SLABS && !packed && img8) {  // (a split image has no ragged tail: numel % 4 == 0)
        img8[e] = static_cast<uint8_t>(
            __nv_cvt_float_to_fp8(static_cast<float>(r), __NV_SATFINITE, __NV_E4M3));
      }
      m[e] = mm;
      v[e] = vv;
    }
    if (packed) Wp[gi] = static_cast<uint8_t>(tern_pack4(pr[0], pr[1], pr[2], pr[3]));
  }
  if (changed) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) n_changed += __shfl_xor_sync(0xffffffffu, n_changed, off);
    if ((threadIdx.x & 31) == 0 && n_changed)
      atomicAdd(changed, static_cast<unsigned long long>(n_changed));
  }
}

__global__ void __launch_bounds__(kThreads)
    slab_sum_kernel(const float* __restrict__ slabs, int nsplit, long long slab,
                    float* __restrict__ out) {
  const int64_t ngroups = slab >> 2;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  for (int64_t gi = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; gi < ngroups;
       gi += stride)
    __stcs(reinterpret_cast<float4*>(out + (gi << 2)), slab_grad4(slabs, nsplit, slab, gi << 2));
  if (blockIdx.x == 0 && threadIdx.x == 0)
    for (int64_t e = ngroups << 2; e < slab; ++e) out[e] = slab_grad1(slabs, nsplit, slab, e);
}

// The deferred last-wave tail of the fused dW GEMM: each thread step takes
// four consecutive columns of one row of a tail tile, sums the token slices'
// partials in slice order, and applies the same update as sr_update_kernel at
// the global element index (so the Philox words are those of the fused path).
// The grid is sized to the blocks that fit at once, and each thread's loads
// for its next group (the optimiser state and the first four slices'
// partials) are issued before it updates the current one.
struct TailGroup {
  float4 p[4];  // partials of slices 0..3
  float4 m, v;
  uint32_t c;   // four int8 codes, or one byte of 2-bit packed codes
  int64_t e;    // first element, or -1 outside the weight
  const float* src;
};

__device__ __forceinline__ void tail_load(int64_t gi, const float* __restrict__ part, int splits,
                                          int tail, int full, int num_n, int M, int N,
                                          const int8_t* __restrict__ W, bool packed,
                                          const float* __restrict__ m, const float* __restrict__ v,
                                          bool col_major, TailGroup& g) {
  const int j = static_cast<int>(gi >> 14);
  const int r = static_cast<int>((gi >> 6) & 255);
  const int c4 = static_cast<int>(gi & 63) * 4;
  const int tile = full + j;
  const int num_m = (M + 255) / 256;  // the GEMM's tile numbering (see its col_major)
  const int row = (col_major ? tile % num_m : tile / num_n) * 256 + r;
  const int col = (col_major ? tile / num_m : tile % num_n) * 256 + c4;
  g.e = -1;
  if (row >= M || col >= N) return;  // N % 4 == 0: the whole group is in range
  g.e = static_cast<int64_t>(row) * N + col;
  if (W) {
    g.m = __ldcs(reinterpret_cast<const float4*>(m + g.e));
    g.v = __ldcs(reinterpret_cast<const float4*>(v + g.e));
    g.c = packed ? static_cast<uint32_t>(reinterpret_cast<const uint8_t*>(W)[g.e >> 2])
                 : *reinterpret_cast<const uint32_t*>(W + g.e);
  }
  g.src = part + static_cast<int64_t>(j) * 65536 + r * 256 + c4;
  const int64_t sstride = static_cast<int64_t>(tail) * 65536;
#pragma unroll
  for (int s = 0; s < 4; ++s)
    if (s < splits) g.p[s] = __ldcs(reinterpret_cast<const float4*>(g.src + s * sstride));
}

template <bool DEV>
__global__ void __launch_bounds__(kThreads, 3)
    tail_update_kernel(const float* __restrict__ part, int splits, int tail, int full, int num_n,
                       int M, int N, int8_t* __restrict__ W, bool packed, float* __restrict__ m,
                       float* __restrict__ v, const UpdateConsts uc_arg,
                       const UpdateConsts* __restrict__ uc_dev, unsigned long long* changed,
                       float* __restrict__ dW_out, const UpdateConsts uc1, int split,
                       bool col_major, uint16_t* __restrict__ img_next,
                       uint8_t* __restrict__ img8_next, bool img8_split) {
  const UpdateConsts uc = DEV ? *uc_dev : uc_arg;
  uint8_t* Wp = reinterpret_cast<uint8_t*>(W);
  const int64_t ngroups = static_cast<int64_t>(tail) * 16384;  // 256 x 256 / 4 per tile
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  const int64_t sstride = static_cast<int64_t>(tail) * 65536;
  uint32_t n_changed = 0;
  int64_t gi = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x;
  TailGroup cur;
  if (gi < ngroups)
    tail_load(gi, part, splits, tail, full, num_n, M, N, W, packed, m, v, col_major, cur);
  for (; gi < ngroups; gi += stride) {
    TailGroup nxt;
    nxt.e = -1;
    if (gi + stride < ngroups)
      tail_load(gi + stride, part, splits, tail, full, num_n, M, N, W, packed, m, v, col_major,
                nxt);
    if (cur.e >= 0) {
      const int64_t e = cur.e;
      float4 g4 = cur.p[0];
#pragma unroll
      for (int s = 1; s < 4; ++s)
        if (s < splits) {
          g4.x = __fadd_rn(g4.x, cur.p[s].x);
          g4.y = __fadd_rn(g4.y, cur.p[s].y);
          g4.z = __fadd_rn(g4.z, cur.p[s].z);
          g4.w = __fadd_rn(g4.w, cur.p[s].w);
        }
      for (int s = 4; s < splits; ++s) {  // slices beyond the fourth, in order
        const float4 h = __ldcs(reinterpret_cast<const float4*>(cur.src + s * sstride));
        g4.x = __fadd_rn(g4.x, h.x);
        g4.y = __fadd_rn(g4.y, h.y);
        g4.z = __fadd_rn(g4.z, h.z);
        g4.w = __fadd_rn(g4.w, h.w);
      }
      if (dW_out) __stcs(reinterpret_cast<float4*>(dW_out + e), g4);
      if (W) {
        const uint32_t craw = cur.c;
        const char4 c0 = packed ? tern_unpack4(craw)
                                : make_char4(static_cast<signed char>(craw & 0xFFu),
                                             static_cast<signed char>((craw >> 8) & 0xFFu),
                                             static_cast<signed char>((craw >> 16) & 0xFFu),
                                             static_cast<signed char>(craw >> 24));
        float4 m4 = cur.m, v4 = cur.v;
        // rows from `split` on: the second of two stacked weights, its own
        // constants and element count
        const bool second = split > 0 && e >= static_cast<int64_t>(split) * N;
        const UpdateConsts& u = second ? uc1 : uc;
        const int64_t er = second ? e - static_cast<int64_t>(split) * N : e;
        uint4 w = make_uint4(0, 0, 0, 0);
        if (u.round_mode == 0)
          w = sr_words(global_blk(u, static_cast<uint64_t>(er >> 2)), u.step_lo, u.tensor_id,
                       u.key0, u.key1);
        const int32_t a = dqt_update_elem(u, g4.x, c0.x, m4.x, v4.x, w.x);
        const int32_t b = dqt_update_elem(u, g4.y, c0.y, m4.y, v4.y, w.y);
        const int32_t c = dqt_update_elem(u, g4.z, c0.z, m4.z, v4.z, w.z);
        const int32_t d = dqt_update_elem(u, g4.w, c0.w, m4.w, v4.w, w.w);
        n_changed += (a != c0.x) + (b != c0.y) + (c != c0.z) + (d != c0.w);
        if (packed)
          Wp[e >> 2] = static_cast<uint8_t>(tern_pack4(a, b, c, d));
        else
          *reinterpret_cast<char4*>(W + e) =
              make_char4(static_cast<signed char>(a), static_cast<signed char>(b),
                         static_cast<signed char>(c), static_cast<signed char>(d));
        if (img_next) {  // the bf16 image of the new codes (exact)
          const __nv_bfloat162 lo = __floats2bfloat162_rn(static_cast<float>(a), static_cast<float>(b));
          const __nv_bfloat162 hi = __floats2bfloat162_rn(static_cast<float>(c), static_cast<float>(d));
          __stcs(reinterpret_cast<uint2*>(img_next + e),
                 make_uint2(*reinterpret_cast<const uint32_t*>(&lo),
                            *reinterpret_cast<const uint32_t*>(&hi)));
        }
        // the E4M3 image of the new codes (exact for |code| <= 16), or their
        // split image (rows of N codes)
        if (img8_next) store_e4m3_4(img8_next, img8_split ? N : 0, e, a, b, c, d);
        __stcs(reinterpret_cast<float4*>(m + e), m4);
        __stcs(reinterpret_cast<float4*>(v + e), v4);
      }
    }
    // the slices' 128-byte lines of these 32 columns (eight lanes' groups)
    // are read: drop them from L2 so that they are never written back
    __syncwarp();
    if ((threadIdx.x & 7) == 0 && cur.e >= 0)
      for (int s = 0; s < splits; ++s)
        asm volatile("discard.global.L2 [%0], 128;" ::"l"(cur.src + s * sstride) : "memory");
    cur = nxt;
  }
  if (changed) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) n_changed += __shfl_xor_sync(0xffffffffu, n_changed, off);
    if ((threadIdx.x & 31) == 0 && n_changed)
      atomicAdd(changed, static_cast<unsigned long long>(n_changed));
  }
}

int stream_blocks(int64_t numel) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t groups = (numel + 3) >> 2;
  int64_t blocks = (groups + kThreads - 1) / kThreads;
  const int64_t cap = static_cast<int64_t>(sms) * 8;  // 8 resident 256-thread blocks per SM
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  return static_cast<int>(blocks);
}

}  // namespace

namespace {

template <bool packed, bool DEV, bool SLABS>
void sr_launch(const float* grad, int splits, long long slab, float* g_out, int8_t* W, float* m,
               float* v, int64_t numel, const UpdateConsts& uc, const UpdateConsts* uc_dev,
               unsigned long long* changed, cudaStream_t stream, uint16_t* img = nullptr,
               uint8_t* img8 = nullptr, int64_t img8_k = 0) {
  sr_update_kernel<packed, DEV, SLABS><<<stream_blocks(numel), kThreads, 0, stream>>>(
      grad, splits, slab, g_out, W, m, v, numel, uc, uc_dev, changed, img, img8, img8_k);
}

template <bool packed>
void sr_dispatch(const float* grad, int splits, long long slab, float* g_out, int8_t* W, float* m,
                 float* v, int64_t numel, const UpdateConsts& uc, const UpdateConsts* uc_dev,
                 unsigned long long* changed, cudaStream_t stream, uint16_t* img = nullptr,
                 uint8_t* img8 = nullptr, int64_t img8_k = 0) {
  // the image outputs are those of the slab instance
  const bool slabs = splits > 1 || g_out || img || img8;
  if (uc_dev) {
    if (slabs)
      sr_launch<packed, true, true>(grad, splits, slab, g_out, W, m, v, numel, uc, uc_dev, changed,
                                    stream, img, img8, img8_k);
    else
      sr_launch<packed, true, false>(grad, 1, 0, nullptr, W, m, v, numel, uc, uc_dev, changed,
                                     stream);
  } else {
    if (slabs)
      sr_launch<packed, false, true>(grad, splits, slab, g_out, W, m, v, numel, uc, nullptr,
                                     changed, stream, img, img8, img8_k);
    else
      sr_launch<packed, false, false>(grad, 1, 0, nullptr, W, m, v, numel, uc, nullptr, changed,
                                      stream);
  }
}

}  // namespace

int launch_sr_update_slabs(const float* slabs, int splits, long long slab, int8_t* W, float* m,
                           float* v, int64_t numel, const UpdateConsts& uc,
                           const UpdateConsts* uc_dev, unsigned long long* changed, float* g_out,
                           cudaStream_t stream, bool packed, uint16_t* img, uint8_t* img8,
                           int64_t img8_k) {
  if (packed)
    sr_dispatch<true>(slabs, splits, slab, g_out, W, m, v, numel, uc, uc_dev, changed, stream);
  else
    sr_dispatch<false>(slabs, splits, slab, g_out, W, m, v, numel, uc, uc_dev, changed, stream,
                       img, img8, img8_k);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_tail_update(const float* part, int splits, int tail, int full, int num_n, int M, int N,
                       int8_t* W, bool packed, float* m, float* v, const UpdateConsts& uc,
                       const UpdateConsts* uc_dev, unsigned long long* changed, float* dW_out,
                       cudaStream_t stream, const UpdateConsts* uc1, int split, bool col_major,
                       uint16_t* img_next, uint8_t* img8_next, bool img8_split) {
  const UpdateConsts u1 = uc1 ? *uc1 : uc;
  // the blocks that fit at once: each thread walks several groups, its next
  // group's loads in flight
  static int occ[2] = {0, 0};  // resident blocks per SM, per template instance
  int& o = occ[uc_dev ? 1 : 0];
  if (o == 0) {
    const void* k = uc_dev ? reinterpret_cast<const void*>(tail_update_kernel<true>)
                           : reinterpret_cast<const void*>(tail_update_kernel<false>);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, k, kThreads, 0) != cudaSuccess || o < 1)
      o = 1;
  }
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (static_cast<int64_t>(tail) * 16384 + kThreads - 1) / kThreads;
  const int64_t cap = static_cast<int64_t>(sms) * o;
  const int blocks = static_cast<int>(want < cap ? want : cap);
  if (uc_dev)
    tail_update_kernel<true><<<blocks, kThreads, 0, stream>>>(part, splits, tail, full, num_n, M, N,
                                                              W, packed, m, v, uc, uc_dev, changed,
                                                              dW_out, u1, uc1 ? split : 0,
                                                              col_major, img_next, img8_next,
                                                              img8_split);
  else
    tail_update_kernel<false><<<blocks, kThreads, 0, stream>>>(part, splits, tail, full, num_n, M,
                                                               N, W, packed, m, v, uc, nullptr,
                                                               changed, dW_out, u1,
                                                               uc1 ? split : 0, col_major,
                                                               img_next, img8_next, img8_split);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_slab_sum(const float* slabs, int splits, long long slab, float* out,
                    cudaStream_t stream) {
  slab_sum_kernel<<<stream_blocks(slab), kThreads, 0, stream>>>(slabs, splits, slab, out);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_sr_update(const float* grad, int8_t* W, float* m, float* v, int64_t numel,
                     const UpdateConsts& uc, const UpdateConsts* uc_dev,
                     unsigned long long* changed, cudaStream_t stream, bool packed) {
  if (packed)
    sr_dispatch<true>(grad, 1, 0, nullptr, W, m, v, numel, uc, uc_dev, changed, stream);
  else
    sr_dispatch<false>(grad, 1, 0, nullptr, W, m, v, numel, uc, uc_dev, changed, stream);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

}  // namespace dqt

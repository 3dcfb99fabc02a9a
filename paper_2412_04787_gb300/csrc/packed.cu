// 2-bit packed ternary storage of DQT weight codes (the ternary footprint of
// Sec. 1: 4 weights per byte instead of 1): conversions between int8 codes and
// packed bytes, and the GEMM operand images (exact bf16 or E4M3 values) built
// straight from the packed bytes.  Code e is field e % 4 (bits 2 (e % 4) and
// 2 (e % 4) + 1) of byte e / 4, a 2-bit two's-complement number; unused fields
// of the last byte are 0.  All kernels are HBM-bound streams; each thread step
// covers 16 codes (4 packed bytes).
#include <cuda_fp8.h>

#include "dqt_internal.h"

namespace dqt {

namespace {

constexpr int kThreads = 256;

int blocks_for(int64_t items) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t b = (items + kThreads - 1) / kThreads;
  const int64_t cap = static_cast<int64_t>(sms) * 8;
  if (b > cap) b = cap;
  return static_cast<int>(b < 1 ? 1 : b);
}

__device__ __forceinline__ uint32_t pack_word(uint32_t w) {  // 4 int8 codes -> 8 bits
  return tern_pack4(static_cast<int8_t>(w & 0xFF), static_cast<int8_t>((w >> 8) & 0xFF),
                    static_cast<int8_t>((w >> 16) & 0xFF), static_cast<int8_t>(w >> 24));
}

__global__ void __launch_bounds__(kThreads)
    pack_kernel(const int8_t* __restrict__ c, int64_t n, uint8_t* __restrict__ out) {
  const int64_t nvec = n >> 4;  // 16 codes -> one 32-bit word of 4 bytes
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; i < nvec;
       i += stride) {
    const uint4 u = __ldcs(reinterpret_cast<const uint4*>(c) + i);
    const uint32_t o = pack_word(u.x) | (pack_word(u.y) << 8) | (pack_word(u.z) << 16) |
                       (pack_word(u.w) << 24);
    reinterpret_cast<uint32_t*>(out)[i] = o;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {  // ragged tail, one thread
    for (int64_t b = nvec * 4; b < (n + 3) / 4; ++b) {
      int32_t f[4] = {0, 0, 0, 0};
      for (int j = 0; j < 4 && 4 * b + j < n; ++j) f[j] = c[4 * b + j];
      out[b] = static_cast<uint8_t>(tern_pack4(f[0], f[1], f[2], f[3]));
    }
  }
}

__global__ void __launch_bounds__(kThreads)
    unpack_kernel(const uint8_t* __restrict__ p, int64_t n, int8_t* __restrict__ c) {
  const int64_t nvec = n >> 4;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; i < nvec;
       i += stride) {
    const uint32_t w = reinterpret_cast<const uint32_t*>(p)[i];
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const char4 q = tern_unpack4((w >> (8 * j)) & 0xFFu);
      o[j] = (static_cast<uint32_t>(static_cast<uint8_t>(q.x))) |
             (static_cast<uint32_t>(static_cast<uint8_t>(q.y)) << 8) |
             (static_cast<uint32_t>(static_cast<uint8_t>(q.z)) << 16) |
             (static_cast<uint32_t>(static_cast<uint8_t>(q.w)) << 24);
    }
    __stcs(reinterpret_cast<uint4*>(c) + i, make_uint4(o[0], o[1], o[2], o[3]));
  }
  if (blockIdx.x == 0 && threadIdx.x == 0)
    for (int64_t e = nvec << 4; e < n; ++e) {
      const char4 q = tern_unpack4(p[e >> 2]);
      const int j = static_cast<int>(e & 3);
      c[e] = j == 0 ? q.x : j == 1 ? q.y : j == 2 ? q.z : q.w;
    }
}

// bf16 bit pattern of a ternary code: -1 -> 0xBF80, 0 -> 0, +1 -> 0x3F80
__device__ __forceinline__ uint32_t tern_bf16(uint32_t f) {
  return f == 1u ? 0x3F80u : (f == 3u ? 0xBF80u : 0u);
}
// E4M3 byte of a ternary code: -1 -> 0xB8, 0 -> 0, +1 -> 0x38
__device__ __forceinline__ uint32_t tern_e4m3(uint32_t f) {
  return f == 1u ? 0x38u : (f == 3u ? 0xB8u : 0u);
}

__global__ void __launch_bounds__(kThreads)
    packed_to_bf16_kernel(const uint8_t* __restrict__ p, int64_t n, uint16_t* __restrict__ img) {
  const int64_t nvec = n >> 4;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; i < nvec;
       i += stride) {
    const uint32_t w = __ldcs(reinterpret_cast<const uint32_t*>(p) + i);
    uint32_t o[8];
#pragma unroll
    for (int j = 0; j < 8; ++j)
      o[j] = tern_bf16((w >> (4 * j)) & 3u) | (tern_bf16((w >> (4 * j + 2)) & 3u) << 16);
    uint4* dst = reinterpret_cast<uint4*>(img) + 2 * i;
    __stcs(dst, make_uint4(o[0], o[1], o[2], o[3]));
    __stcs(dst + 1, make_uint4(o[4], o[5], o[6], o[7]));
  }
  if (blockIdx.x == 0 && threadIdx.x == 0)
    for (int64_t e = nvec << 4; e < n; ++e)
      img[e] = static_cast<uint16_t>(tern_bf16((p[e >> 2] >> (2 * (e & 3))) & 3u));
}

__global__ void __launch_bounds__(kThreads)
    packed_to_fp8_kernel(const uint8_t* __restrict__ p, int64_t n, uint8_t* __restrict__ out) {
  const int64_t nvec = n >> 4;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; i < nvec;
       i += stride) {
    const uint32_t w = __ldcs(reinterpret_cast<const uint32_t*>(p) + i);
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
      o[j] = tern_e4m3((w >> (8 * j)) & 3u) | (tern_e4m3((w >> (8 * j + 2)) & 3u) << 8) |
             (tern_e4m3((w >> (8 * j + 4)) & 3u) << 16) |
             (tern_e4m3((w >> (8 * j + 6)) & 3u) << 24);
    __stcs(reinterpret_cast<uint4*>(out) + i, make_uint4(o[0], o[1], o[2], o[3]));
  }
  if (blockIdx.x == 0 && threadIdx.x == 0)
    for (int64_t e = nvec << 4; e < n; ++e)
      out[e] = static_cast<uint8_t>(tern_e4m3((p[e >> 2] >> (2 * (e & 3))) & 3u));
}

}  // namespace

int launch_pack_ternary(const int8_t* c, int64_t n, uint8_t* out, cudaStream_t stream) {
  pack_kernel<<<blocks_for(n >> 4), kThreads, 0, stream>>>(c, n, out);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_unpack_ternary(const uint8_t* p, int64_t n, int8_t* c, cudaStream_t stream) {
  unpack_kernel<<<blocks_for(n >> 4), kThreads, 0, stream>>>(p, n, c);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_packed_to_bf16(const uint8_t* p, int64_t n, uint16_t* img, cudaStream_t stream) {
  packed_to_bf16_kernel<<<blocks_for(n >> 4), kThreads, 0, stream>>>(p, n, img);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_packed_to_fp8(const uint8_t* p, int64_t n, uint8_t* out, cudaStream_t stream) {
  packed_to_fp8_kernel<<<blocks_for(n >> 4), kThreads, 0, stream>>>(p, n, out);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

}  // namespace dqt

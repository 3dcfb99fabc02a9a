// Bandwidth-bound quantisation kernels of a DQT BitLinear step:
//   act_quant      8-bit per-token absmax activation codes (Sec. 3.2) plus the
//                  bf16 operand images the tensor-core GEMMs read
//   codes_to_bf16  exact bf16 image of the int8 weight codes
//   absmean_*      Eq. 2-4 initialisation (deterministic fp64 reduction)
// and, for the FP8 environment (Sec. 4.1/4.3), the same activation kernels
// emitting E4M3 bytes with the per-token scale 448 / max(amax, 1e-5) (template
// flag F8), and the E4M3 image of the weight codes.
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include "dqt_internal.h"

namespace dqt {

namespace {

__device__ __forceinline__ float bf16_bits_to_f32(uint32_t h) { return __uint_as_float(h << 16); }

__device__ __forceinline__ uint16_t f32_to_bf16_bits(float f) {
  const __nv_bfloat16 h = __float2bfloat16_rn(f);
  return *reinterpret_cast<const uint16_t*>(&h);
}

// The 8-bit activation code of eight bf16 values (one 16-byte vector) at
// scale s: int8 Clip[Round(x s), -128, 127], or (F8) the E4M3 byte of x s,
// round-to-nearest-even with saturation.  Each product is one fp32 multiply.
template <bool F8>
__device__ __forceinline__ void quant8(const uint4 u, float s, int32_t (&q)[8]) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float lo = __fmul_rn(bf16_bits_to_f32(w[j] & 0xFFFFu), s);
    const float hi = __fmul_rn(bf16_bits_to_f32(w[j] >> 16), s);
    if (F8) {
      const uint32_t b = __nv_cvt_float2_to_fp8x2(make_float2(lo, hi), __NV_SATFINITE, __NV_E4M3);
      q[2 * j] = static_cast<int32_t>(b & 0xFFu);
      q[2 * j + 1] = static_cast<int32_t>((b >> 8) & 0xFFu);
    } else {
      q[2 * j] = static_cast<int32_t>(fminf(fmaxf(rintf(lo), -128.0f), 127.0f));
      q[2 * j + 1] = static_cast<int32_t>(fminf(fmaxf(rintf(hi), -128.0f), 127.0f));
    }
  }
}

template <bool F8>
__device__ __forceinline__ float code_scale_num() { return F8 ? 448.0f : 127.0f; }

// Entry j of the dequantisation table: bf16(value / s) for the code whose
// table index is j (int8 code j - 128, or E4M3 byte j).
template <bool F8>
__device__ __forceinline__ uint16_t dq_entry(int j, float s) {
  float v;
  if (F8) {
    const __half h(__nv_cvt_fp8_to_halfraw(static_cast<__nv_fp8_storage_t>(j), __NV_E4M3));
    v = __half2float(h);
  } else {
    v = static_cast<float>(j - 128);
  }
  return f32_to_bf16_bits(__fdiv_rn(v, s));
}

template <bool F8>
__device__ __forceinline__ int dq_index(int32_t q) { return F8 ? q : q + 128; }

// One warp per token row; 16-byte (8 x bf16) vector accesses.  Pass 1 finds
// amax; pass 2 re-reads the row (an L1/L2 hit) and writes the outputs.
constexpr int kAqWarps = 8;

template <bool F8>
__global__ void __launch_bounds__(kAqWarps * 32)
    act_quant_kernel(const uint16_t* __restrict__ X, int T, int K, int8_t* __restrict__ Xq,
                     float* __restrict__ s_x, uint16_t* __restrict__ Xq_img,
                     uint16_t* __restrict__ Xdq) {
  const int row = blockIdx.x * kAqWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= T) return;
  const int nv = K >> 3;
  const uint4* xr = reinterpret_cast<const uint4*>(X + static_cast<size_t>(row) * K);

  float amax = 0.0f;
#pragma unroll 4
  for (int i = lane; i < nv; i += 32) {
    const uint4 u = __ldg(xr + i);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      amax = fmaxf(amax, fabsf(bf16_bits_to_f32(w[j] & 0xFFFFu)));
      amax = fmaxf(amax, fabsf(bf16_bits_to_f32(w[j] >> 16)));
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
  const float s = __fdiv_rn(code_scale_num<F8>(), fmaxf(amax, 1e-5f));
  if (lane == 0) s_x[row] = s;

  const size_t rbase = static_cast<size_t>(row) * K;
#pragma unroll 4
  for (int i = lane; i < nv; i += 32) {
    const uint4 u = __ldg(xr + i);
    int32_t q[8];
    quant8<F8>(u, s, q);
    const size_t e = rbase + static_cast<size_t>(i) * 8;
    if (Xq) {
      uint2 pk;
      pk.x = (q[0] & 0xFF) | ((q[1] & 0xFF) << 8) | ((q[2] & 0xFF) << 16) | ((q[3] & 0xFF) << 24);
      pk.y = (q[4] & 0xFF) | ((q[5] & 0xFF) << 8) | ((q[6] & 0xFF) << 16) | ((q[7] & 0xFF) << 24);
      *reinterpret_cast<uint2*>(Xq + e) = pk;
    }
    if (Xq_img) {
      uint4 pk;
      pk.x = f32_to_bf16_bits(static_cast<float>(q[0])) | (uint32_t(f32_to_bf16_bits(static_cast<float>(q[1]))) << 16);
      pk.y = f32_to_bf16_bits(static_cast<float>(q[2])) | (uint32_t(f32_to_bf16_bits(static_cast<float>(q[3]))) << 16);
      pk.z = f32_to_bf16_bits(static_cast<float>(q[4])) | (uint32_t(f32_to_bf16_bits(static_cast<float>(q[5]))) << 16);
      pk.w = f32_to_bf16_bits(static_cast<float>(q[6])) | (uint32_t(f32_to_bf16_bits(static_cast<float>(q[7]))) << 16);
      *reinterpret_cast<uint4*>(Xq_img + e) = pk;
    }
    if (Xdq) {
      uint32_t h[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) h[j] = dq_entry<F8>(dq_index<F8>(q[j]), s);
      uint4 pk;
      pk.x = h[0] | (h[1] << 16);
      pk.y = h[2] | (h[3] << 16);
      pk.z = h[4] | (h[5] << 16);
      pk.w = h[6] | (h[7] << 16);
      *reinterpret_cast<uint4*>(Xdq + e) = pk;
    }
  }
}

// Activation quantisation with whole rows staged in shared memory: one CTA
// per SM, a producer lane that streams the CTA's rows (blockIdx.x,
// blockIdx.x + gridDim.x, ...) with linear bulk copies into a ring of S row
// slots, and W consumer warps, warp w owning slots w, w + W, ... (S a
// multiple of W, at least two slots per warp).  The j-th row of the CTA goes
// to slot j % S and is processed by one warp: pass 1 reduces amax over the
// row in shared memory, pass 2 re-reads it and writes the outputs.  Every
// slot carries a `full` barrier (the copy's bytes) and an `empty` barrier
// (one arrive by its consumer warp); the ring keeps up to S rows in flight
// per SM, which a register-held design cannot.
//
// amax is reduced on pairs of bf16 magnitudes (max.bf16x2 returns the
// non-NaN operand, as fmaxf does, and is exact).  Round(y) for the int8
// codes is taken with the fp32 add y + 1.5 * 2^23, which rounds to the
// nearest integer, half to even, for |y| < 2^22; the code is then the low
// byte of the sum's bit pattern.  Here y = RN(x s) with |x| <= a and
// s = RN(127 / a), a = max(amax, 1e-5), so |y| <= RN(127 (1 + 2^-24)) <=
// 127 + 2^-17 and the sum never exceeds 1.5 * 2^23 + 127: only the lower
// clamp is needed, and it maps a NaN product (an infinite input) to -128, as
// act_quant_kernel does.
constexpr int kAqbRing = 192 * 1024;  // shared-memory bytes of the row ring

// Linear bulk copy (no tensor map) of `bytes` from global memory into this
// CTA's shared memory, completing on `bar`, whose expected byte count the
// caller has raised by `bytes`.  Both addresses 16-byte aligned; `bytes` a
// multiple of 16.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes,
                                          uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// The ring of row chunks in dynamic shared memory: S slots of rpc rows of
// row_bytes, then S `full` and S `empty` mbarriers.  CTA b owns the rows
// [b T / G, (b + 1) T / G) (G = gridDim.x <= T, so at least one), cut into
// chunks of rpc rows (the last one shorter); chunk j is one linear bulk copy
// into slot j % S and is processed by consumer warp j % W (S a multiple of W).
struct RowRing {
  uint8_t* base;
  uint64_t* full;
  uint64_t* empty;
  uint32_t row_bytes;
  int S, rpc;
  int64_t lo, hi;  // this CTA's rows
  int nchunks;

  __device__ __forceinline__ RowRing(uint8_t* smem, int slots, uint32_t rb, int rows_per_chunk,
                                     int64_t T)
      : base(smem),
        full(reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(slots) * rows_per_chunk * rb)),
        empty(full + slots),
        row_bytes(rb),
        S(slots),
        rpc(rows_per_chunk),
        lo(static_cast<int64_t>(blockIdx.x) * T / gridDim.x),
        hi(static_cast<int64_t>(blockIdx.x + 1) * T / gridDim.x) {
    nchunks = static_cast<int>((hi - lo + rpc - 1) / rpc);
  }
  // shared memory after the ring and its barriers
  __device__ __forceinline__ uint8_t* end() const { return reinterpret_cast<uint8_t*>(empty + S); }

  // every thread, followed by __syncthreads()
  __device__ __forceinline__ void init_barriers() const {
    if (static_cast<int>(threadIdx.x) < S) {
      mbar_init(&full[threadIdx.x], 1);
      mbar_init(&empty[threadIdx.x], 1);
      fence_mbarrier_init();
    }
  }

  __device__ __forceinline__ int64_t row0(int j) const { return lo + static_cast<int64_t>(j) * rpc; }
  __device__ __forceinline__ int rows(int j) const {
    const int64_t r = hi - row0(j);
    return r < rpc ? static_cast<int>(r) : rpc;
  }

  // One thread: the chunks of this CTA from `src` (rows of row_bytes bytes),
  // each slot refilled once its consumer has released it; returns when every
  // copy it issued has landed (the CTA must not retire before).
  __device__ void produce(const uint8_t* src, unsigned int* status, uint64_t limit_ns) const {
    int issued = 0;
    for (; issued < nchunks; ++issued) {
      const int slot = issued % S, use = issued / S;
      if (use > 0 && !mbar_wait(&empty[slot], (use - 1) & 1, limit_ns)) {
        record_timeout(status);
        break;
      }
      const uint32_t bytes = static_cast<uint32_t>(rows(issued)) * row_bytes;
      mbar_arrive_expect_tx(&full[slot], bytes);
      bulk_load(base + static_cast<size_t>(slot) * rpc * row_bytes,
                src + static_cast<size_t>(row0(issued)) * row_bytes, bytes, &full[slot]);
    }
    for (int j = issued > S ? issued - S : 0; j < issued; ++j)
      if (!mbar_wait(&full[j % S], (j / S) & 1, limit_ns)) {
        record_timeout(status);
        break;
      }
  }

  // All lanes of the consumer warp: waits for chunk j; false (warp-uniform,
  // timeout recorded) if it did not arrive in time.
  __device__ __forceinline__ bool acquire(int j, int lane, unsigned int* status,
                                          uint64_t limit_ns) const {
    const bool ok = __all_sync(0xffffffffu, mbar_wait(&full[j % S], (j / S) & 1, limit_ns));
    if (!ok && lane == 0) record_timeout(status);
    return ok;
  }
  // row r of chunk j
  __device__ __forceinline__ const uint8_t* row(int j, int r) const {
    return base + (static_cast<size_t>(j % S) * rpc + r) * row_bytes;
  }
  // All lanes, after their last read of the slot.
  __device__ __forceinline__ void release(int j, int lane) const {
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[j % S]);
  }
};

template <bool F8>
__global__ void __launch_bounds__(32 * 17, 1)
    act_quant_bulk_kernel(const uint16_t* __restrict__ X, int T, int K,
                          int8_t* __restrict__ Xq, float* __restrict__ s_x,
                          uint16_t* __restrict__ Xq_img, uint16_t* __restrict__ Xdq, int S, int W,
                          int rpc, unsigned int* status, uint64_t limit_ns) {
  extern __shared__ __align__(128) uint8_t aqb_smem[];
  const RowRing ring(aqb_smem, S, static_cast<uint32_t>(K) * 2u, rpc, T);
  uint16_t* tables = reinterpret_cast<uint16_t*>(ring.end());
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  ring.init_barriers();
  __syncthreads();
  if (warp == 0) {
    if (lane == 0) ring.produce(reinterpret_cast<const uint8_t*>(X), status, limit_ns);
    return;
  }

  const int cw = warp - 1;
  uint16_t* table = tables + cw * 256;
  const int nv = K >> 3;  // 16-byte vectors per row
  constexpr float kMagic = 12582912.0f;  // 1.5 * 2^23
  for (int j = cw; j < ring.nchunks; j += W) {
    if (!ring.acquire(j, lane, status, limit_ns)) return;
    const int nr = ring.rows(j);
#pragma unroll 1
    for (int r = 0; r < nr; ++r) {
      const int64_t row = ring.row0(j) + r;
      const uint4* xr = reinterpret_cast<const uint4*>(ring.row(j, r));
      __nv_bfloat162 am2 = __floats2bfloat162_rn(0.0f, 0.0f);
#pragma unroll 4
      for (int v = lane; v < nv; v += 32) {
        const uint4 u = xr[v];
        const uint32_t w[4] = {u.x & 0x7FFF7FFFu, u.y & 0x7FFF7FFFu, u.z & 0x7FFF7FFFu,
                               u.w & 0x7FFF7FFFu};
#pragma unroll
        for (int i = 0; i < 4; ++i) am2 = __hmax2(am2, *reinterpret_cast<const __nv_bfloat162*>(&w[i]));
      }
      float amax = fmaxf(__low2float(am2), __high2float(am2));
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
      const float s = __fdiv_rn(code_scale_num<F8>(), fmaxf(amax, 1e-5f));
      if (lane == 0) s_x[row] = s;
      if (Xdq) {
        for (int i = lane; i < 256; i += 32) table[i] = dq_entry<F8>(i, s);
        __syncwarp();
      }
      const size_t rbase = static_cast<size_t>(row) * K;
#pragma unroll 4
      for (int v = lane; v < nv; v += 32) {
        const uint4 u = xr[v];
        const size_t e = rbase + static_cast<size_t>(v) * 8;
        uint32_t b[8];  // per element: the code's table index in the low byte
        if (F8) {
          int32_t q[8];
          quant8<true>(u, s, q);
#pragma unroll
          for (int i = 0; i < 8; ++i) b[i] = static_cast<uint32_t>(q[i]);
        } else {
          const uint32_t w[4] = {u.x, u.y, u.z, u.w};
          float z[8];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            z[2 * i] = __fadd_rn(__fmul_rn(bf16_bits_to_f32(w[i] & 0xFFFFu), s), kMagic);
            z[2 * i + 1] = __fadd_rn(__fmul_rn(bf16_bits_to_f32(w[i] >> 16), s), kMagic);
          }
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            z[i] = fmaxf(z[i], kMagic - 128.0f);
            b[i] = __float_as_uint(z[i]);
          }
          if (Xq_img) {
            uint32_t h[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const __nv_bfloat162 p =
                  __floats2bfloat162_rn(__fsub_rn(z[2 * i], kMagic), __fsub_rn(z[2 * i + 1], kMagic));
              h[i] = *reinterpret_cast<const uint32_t*>(&p);
            }
            __stcs(reinterpret_cast<uint4*>(Xq_img + e), make_uint4(h[0], h[1], h[2], h[3]));
          }
        }
        if (Xq) {
          uint2 pk;
          pk.x = __byte_perm(__byte_perm(b[0], b[1], 0x0040), __byte_perm(b[2], b[3], 0x0040), 0x5410);
          pk.y = __byte_perm(__byte_perm(b[4], b[5], 0x0040), __byte_perm(b[6], b[7], 0x0040), 0x5410);
          __stcs(reinterpret_cast<uint2*>(Xq + e), pk);
        }
        if (Xdq) {
          uint32_t h[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) h[i] = table[F8 ? (b[i] & 0xFFu) : ((b[i] & 0xFFu) ^ 0x80u)];
          __stcs(reinterpret_cast<uint4*>(Xdq + e),
                 make_uint4(h[0] | (h[1] << 16), h[2] | (h[3] << 16), h[4] | (h[5] << 16),
                            h[6] | (h[7] << 16)));
        }
      }
      __syncwarp();  // the table is rewritten for the next row
    }
    ring.release(j, lane);  // the slot is read for the last time
  }
}

// X_tilde = bf16(q / s_x) from int8 activation codes (the dW operand of the
// int8 call), rows staged as in act_quant_bulk_kernel: each consumer warp
// builds its row's 256-entry table of correctly rounded quotients (the table
// dqt_act_quant uses), then maps the row's codes through it, 16 codes (one
// 16-byte shared load, two 16-byte stores) per lane step.  K % 16 == 0.
__global__ void __launch_bounds__(32 * 17, 1)
    codes_to_xdq_bulk_kernel(const int8_t* __restrict__ Xq, const float* __restrict__ s_x, int T,
                             int K, uint16_t* __restrict__ Xdq, int S, int W, int rpc,
                             unsigned int* status, uint64_t limit_ns) {
  extern __shared__ __align__(128) uint8_t cxb_smem[];
  const RowRing ring(cxb_smem, S, static_cast<uint32_t>(K), rpc, T);
  uint16_t* tables = reinterpret_cast<uint16_t*>(ring.end());
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  ring.init_barriers();
  __syncthreads();
  if (warp == 0) {
    if (lane == 0) ring.produce(reinterpret_cast<const uint8_t*>(Xq), status, limit_ns);
    return;
  }
  const int cw = warp - 1;
  uint16_t* t = tables + cw * 256;
  const int nv = K >> 4;
  for (int j = cw; j < ring.nchunks; j += W) {
    const int nr = ring.rows(j);
    bool acquired = false;
#pragma unroll 1
    for (int r = 0; r < nr; ++r) {
      const int64_t row = ring.row0(j) + r;
      const float s = s_x[row];
#pragma unroll
      for (int i = lane; i < 256; i += 32) t[i] = dq_entry<false>(i, s);
      __syncwarp();
      if (!acquired) {
        if (!ring.acquire(j, lane, status, limit_ns)) return;
        acquired = true;
      }
      const uint4* src = reinterpret_cast<const uint4*>(ring.row(j, r));
      uint4* dst = reinterpret_cast<uint4*>(Xdq + static_cast<size_t>(row) * K);
#pragma unroll 4
      for (int v = lane; v < nv; v += 32) {
        const uint4 u = src[v];
        const uint32_t w[4] = {u.x ^ 0x80808080u, u.y ^ 0x80808080u, u.z ^ 0x80808080u,
                               u.w ^ 0x80808080u};  // table indices q + 128
        uint32_t h[8];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          h[2 * i] = t[w[i] & 0xFFu] | (uint32_t(t[(w[i] >> 8) & 0xFFu]) << 16);
          h[2 * i + 1] = t[(w[i] >> 16) & 0xFFu] | (uint32_t(t[w[i] >> 24]) << 16);
        }
        __stcs(dst + 2 * v, make_uint4(h[0], h[1], h[2], h[3]));
        __stcs(dst + 2 * v + 1, make_uint4(h[4], h[5], h[6], h[7]));
      }
      __syncwarp();  // the table is rewritten for the next row
    }
    ring.release(j, lane);  // the slot is read for the last time
  }
}

// X_tilde = bf16(q / s_x) from int8 activation codes: the operand the
// weight-gradient GEMM reads.  One warp per token row; the row's 256 possible
// values come from a per-warp table of correctly rounded fp32 divisions (the
// table dqt_act_quant uses), so the image is bit-identical to the one it
// writes.  16 codes (one 16-byte load, two 16-byte stores) per lane step;
// K % 16 == 0.
__global__ void __launch_bounds__(256)
    codes_to_xdq_kernel(const int8_t* __restrict__ Xq, const float* __restrict__ s_x, int T,
                        int K, uint16_t* __restrict__ Xdq) {
  __shared__ uint16_t table[8][256];
  const int wid = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nv = K >> 4;
  for (int row = blockIdx.x * 8 + wid; row < T; row += gridDim.x * 8) {
    const float s = s_x[row];
    __syncwarp();  // the previous row's lookups are done
#pragma unroll
    for (int j = lane; j < 256; j += 32) table[wid][j] = dq_entry<false>(j, s);
    __syncwarp();
    const uint4* src = reinterpret_cast<const uint4*>(Xq + static_cast<size_t>(row) * K);
    uint4* dst = reinterpret_cast<uint4*>(Xdq + static_cast<size_t>(row) * K);
    for (int v = lane; v < nv; v += 32) {
      const uint4 u = __ldcs(src + v);
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
      uint32_t h[8];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint16_t* t = table[wid];
        h[2 * j] = t[((w[j] & 0xFFu) ^ 0x80u)] | (uint32_t(t[((w[j] >> 8) & 0xFFu) ^ 0x80u]) << 16);
        h[2 * j + 1] =
            t[((w[j] >> 16) & 0xFFu) ^ 0x80u] | (uint32_t(t[(w[j] >> 24) ^ 0x80u]) << 16);
      }
      __stcs(dst + 2 * v, make_uint4(h[0], h[1], h[2], h[3]));
      __stcs(dst + 2 * v + 1, make_uint4(h[4], h[5], h[6], h[7]));
    }
  }
}

// 64 codes per thread per step: four 16-byte loads issued together, then
// eight 16-byte streaming stores (the image is read by the next kernel only).
__device__ __forceinline__ void codes16_to_bf16(const uint4 u, uint4& o0, uint4& o1) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
  uint32_t o[8];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int32_t b0 = static_cast<int8_t>(w[j] & 0xFF);
    const int32_t b1 = static_cast<int8_t>((w[j] >> 8) & 0xFF);
    const int32_t b2 = static_cast<int8_t>((w[j] >> 16) & 0xFF);
    const int32_t b3 = static_cast<int8_t>(w[j] >> 24);
    o[2 * j] = f32_to_bf16_bits(static_cast<float>(b0)) |
               (uint32_t(f32_to_bf16_bits(static_cast<float>(b1))) << 16);
    o[2 * j + 1] = f32_to_bf16_bits(static_cast<float>(b2)) |
                   (uint32_t(f32_to_bf16_bits(static_cast<float>(b3))) << 16);
  }
  o0 = make_uint4(o[0], o[1], o[2], o[3]);
  o1 = make_uint4(o[4], o[5], o[6], o[7]);
}

__global__ void codes_to_bf16_kernel(const int8_t* __restrict__ W, int64_t numel,
                                     uint16_t* __restrict__ img) {
  const int64_t nvec = numel >> 4;  // 16-code vectors
  const int64_t nthr = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const uint4* src = reinterpret_cast<const uint4*>(W);
  uint4* dst = reinterpret_cast<uint4*>(img);
  const int64_t t0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  // groups of four vectors, consecutive threads on consecutive vectors
  for (int64_t base = 0; base < nvec; base += 4 * nthr) {
    uint4 u[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t i = base + j * nthr + t0;
      u[j] = i < nvec ? __ldcs(src + i) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t i = base + j * nthr + t0;
      if (i < nvec) {
        uint4 o0, o1;
        codes16_to_bf16(u[j], o0, o1);
        __stcs(dst + 2 * i, o0);
        __stcs(dst + 2 * i + 1, o1);
      }
    }
  }
  // ragged tail (numel % 16 elements), one thread
  if (blockIdx.x == 0 && threadIdx.x == 0)
    for (int64_t e = nvec << 4; e < numel; ++e) img[e] = f32_to_bf16_bits(static_cast<float>(W[e]));
}

// E4M3 image of weight codes of magnitude <= 16 (exact): 16 codes per thread.
__device__ __forceinline__ uint32_t codes4_to_e4m3(uint32_t w) {
  const float c0 = static_cast<float>(static_cast<int8_t>(w & 0xFF));
  const float c1 = static_cast<float>(static_cast<int8_t>((w >> 8) & 0xFF));
  const float c2 = static_cast<float>(static_cast<int8_t>((w >> 16) & 0xFF));
  const float c3 = static_cast<float>(static_cast<int8_t>(w >> 24));
  const uint32_t lo = __nv_cvt_float2_to_fp8x2(make_float2(c0, c1), __NV_SATFINITE, __NV_E4M3);
  const uint32_t hi = __nv_cvt_float2_to_fp8x2(make_float2(c2, c3), __NV_SATFINITE, __NV_E4M3);
  return (lo & 0xFFFFu) | ((hi & 0xFFFFu) << 16);
}

__global__ void codes_to_fp8_kernel(const int8_t* __restrict__ W, int64_t numel,
                                    uint8_t* __restrict__ out) {
  const int64_t nvec = numel >> 4;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const uint4* src = reinterpret_cast<const uint4*>(W);
  uint4* dst = reinterpret_cast<uint4*>(out);
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec;
       i += stride) {
    const uint4 u = __ldcs(src + i);
    __stcs(dst + i, make_uint4(codes4_to_e4m3(u.x), codes4_to_e4m3(u.y), codes4_to_e4m3(u.z),
                               codes4_to_e4m3(u.w)));
  }
  if (blockIdx.x == 0 && threadIdx.x == 0)
    for (int64_t e = nvec << 4; e < numel; ++e)
      out[e] = static_cast<uint8_t>(codes4_to_e4m3(static_cast<uint8_t>(W[e])) & 0xFFu);
}

// E4M3 split image of codes wider than 16 in magnitude: c = 16 h + l with
// h = c >> 4 (floor(c / 16), in [-8, 7]) and l = c & 15 (in [0, 15]); 16 h
// (a multiple of 16 of magnitude <= 128, at most three significant bits)
// and l are E4M3 values, so each half is exact.  Row n of the [N, 2K] image:
// 16 h of its K codes, then their l.  One thread step: 16 codes of a row.
__global__ void codes_to_fp8_split_kernel(const int8_t* __restrict__ W, int64_t N, int64_t K,
                                          uint8_t* __restrict__ out) {
  const int64_t vpr = K >> 4;  // 16-code vectors per row
  const int64_t nvec = N * vpr;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec;
       i += stride) {
    const int64_t n = i / vpr, k = (i - n * vpr) << 4;
    const uint4 u = __ldcs(reinterpret_cast<const uint4*>(W + n * K + k));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
    uint32_t hi[4], lo[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      float h[4], l[4];
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const int32_t c = static_cast<int8_t>((w[j] >> (8 * b)) & 0xFFu);
        h[b] = static_cast<float>(16 * (c >> 4));
        l[b] = static_cast<float>(c & 15);
      }
      const uint32_t h01 = __nv_cvt_float2_to_fp8x2(make_float2(h[0], h[1]), __NV_SATFINITE, __NV_E4M3);
      const uint32_t h23 = __nv_cvt_float2_to_fp8x2(make_float2(h[2], h[3]), __NV_SATFINITE, __NV_E4M3);
      const uint32_t l01 = __nv_cvt_float2_to_fp8x2(make_float2(l[0], l[1]), __NV_SATFINITE, __NV_E4M3);
      const uint32_t l23 = __nv_cvt_float2_to_fp8x2(make_float2(l[2], l[3]), __NV_SATFINITE, __NV_E4M3);
      hi[j] = (h01 & 0xFFFFu) | ((h23 & 0xFFFFu) << 16);
      lo[j] = (l01 & 0xFFFFu) | ((l23 & 0xFFFFu) << 16);
    }
    uint8_t* row = out + n * 2 * K;
    __stcs(reinterpret_cast<uint4*>(row + k), make_uint4(hi[0], hi[1], hi[2], hi[3]));
    __stcs(reinterpret_cast<uint4*>(row + K + k), make_uint4(lo[0], lo[1], lo[2], lo[3]));
  }
}

// Eq. 2, stage 1: each of kAbsmeanBlocks blocks sums |w| in fp64 over a fixed
// strided subset and reduces in a fixed tree: the result does not depend on
// scheduling.
constexpr int kAbsThreads = 256;

__global__ void __launch_bounds__(kAbsThreads)
    absmean_partial_kernel(const float* __restrict__ W0, int64_t numel, double* __restrict__ ws) {
  __shared__ double sh[kAbsThreads];
  const int64_t stride = static_cast<int64_t>(kAbsmeanBlocks) * kAbsThreads;
  double acc = 0.0;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kAbsThreads + threadIdx.x; i < numel;
       i += stride)
    acc += fabs(static_cast<double>(W0[i]));
  sh[threadIdx.x] = acc;
  __syncthreads();
  for (int w = kAbsThreads / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) sh[threadIdx.x] += sh[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) ws[blockIdx.x] = sh[0];
}

// Eq. 2, stage 2: one block reduces the kAbsmeanBlocks partials, fixed tree.
__global__ void __launch_bounds__(kAbsmeanBlocks) absmean_final_kernel(double* ws) {
  __shared__ double sh[kAbsmeanBlocks];
  sh[threadIdx.x] = ws[threadIdx.x];
  __syncthreads();
  for (int w = kAbsmeanBlocks / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) sh[threadIdx.x] += sh[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) ws[kAbsmeanBlocks] = sh[0];
}

// Eq. 4: codes = Clip[Round(W0 * s_w), qmin, qmax], fp32 multiply, half-to-even.
__global__ void absmean_codes_kernel(const float* __restrict__ W0, int64_t numel, float s,
                                     int32_t qmin, int32_t qmax, int8_t* __restrict__ codes) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < numel;
       i += stride) {
    const float r = rintf(__fmul_rn(W0[i], s));
    const float c = fminf(fmaxf(r, static_cast<float>(qmin)), static_cast<float>(qmax));
    codes[i] = static_cast<int8_t>(static_cast<int32_t>(c));
  }
}

int grid_for(int64_t work, int threads) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (work + threads - 1) / threads;
  const int64_t cap = static_cast<int64_t>(sms) * 8;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

}  // namespace

namespace {

// Geometry of a row ring (act_quant_bulk_kernel, codes_to_xdq_bulk_kernel):
// chunks of about 8 KB (rows of up to 8 KB are copied one per chunk), then up
// to 16 consumer warps and as many slots per warp as fit in kAqbRing bytes
// (48 slots at most); false when fewer than four chunks fit.  One producer
// thread issues a bulk copy about every 0.2 us whatever its size, so copies
// below ~8 KB leave the ring short of bytes in flight.
bool ring_geometry(int64_t row_bytes, int& rpc, int& W, int& S) {
  rpc = row_bytes >= 8192 ? 1 : static_cast<int>(8192 / row_bytes);
  const int64_t smax = kAqbRing / (rpc * row_bytes);
  if (smax < 4) return false;
  W = static_cast<int>(smax < 16 ? smax : 16);
  S = static_cast<int>(smax < 48 ? smax : 48) / W * W;
  return true;
}
constexpr int kRingMaxSmem = kAqbRing + 16 * 48 + 16 * 512;  // ring, barriers, tables

// Launches a row-ring kernel: one CTA per SM (at most T), 32 (W + 1) threads.
template <typename Kern, typename... Args>
int launch_ring(Kern kern, bool& attr_set, int64_t T, int rpc, int W, int S, int64_t row_bytes,
                cudaStream_t stream, Args... args) {
  if (!attr_set) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kRingMaxSmem) !=
        cudaSuccess)
      return 3;
    attr_set = true;
  }
  unsigned int* status = status_word();
  if (!status) return 3;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int blocks = static_cast<int>(T < sms ? T : sms);
  const size_t smem =
      static_cast<size_t>(S) * rpc * row_bytes + 16 * static_cast<size_t>(S) + 512 * W;
  kern<<<blocks, 32 * (W + 1), smem, stream>>>(args..., S, W, rpc, status, wait_limit_ns());
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

// Rows staged in shared memory when at least four fit in the ring; -1 when
// the rows are too long.
template <bool F8>
int launch_aq_bulk(const uint16_t* X, int64_t T, int64_t K, int8_t* Xq, float* s_x,
                   uint16_t* Xq_img, uint16_t* Xdq, cudaStream_t stream) {
  int rpc, W, S;
  if (!ring_geometry(2 * K, rpc, W, S)) return -1;
  static bool attr_set = false;  // per template instance
  return launch_ring(act_quant_bulk_kernel<F8>, attr_set, T, rpc, W, S, 2 * K, stream, X,
                     static_cast<int>(T), static_cast<int>(K), Xq, s_x, Xq_img, Xdq);
}

template <bool F8>
int launch_aq(const uint16_t* X, int64_t T, int64_t K, int8_t* Xq, float* s_x, uint16_t* Xq_img,
              uint16_t* Xdq, cudaStream_t stream) {
  {
    const int r = launch_aq_bulk<F8>(X, T, K, Xq, s_x, Xq_img, Xdq, stream);
    if (r >= 0) return r;
  }
  // rows longer than 48 KB (K > 24576): one warp per row, two passes
  const int blocks = static_cast<int>((T + kAqWarps - 1) / kAqWarps);
  act_quant_kernel<F8><<<blocks, kAqWarps * 32, 0, stream>>>(X, static_cast<int>(T),
                                                            static_cast<int>(K), Xq, s_x, Xq_img, Xdq);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

}  // namespace

int launch_act_quant(const uint16_t* X, int64_t T, int64_t K, int8_t* Xq, float* s_x,
                     uint16_t* Xq_img, uint16_t* Xdq, cudaStream_t stream) {
  return launch_aq<false>(X, T, K, Xq, s_x, Xq_img, Xdq, stream);
}

int launch_codes_to_xdq(const int8_t* Xq, const float* s_x, int64_t T, int64_t K, uint16_t* Xdq,
                        cudaStream_t stream) {
  {
    int rpc, W, S;
    if (ring_geometry(K, rpc, W, S)) {
      static bool attr_set = false;
      return launch_ring(codes_to_xdq_bulk_kernel, attr_set, T, rpc, W, S, K, stream, Xq, s_x,
                         static_cast<int>(T), static_cast<int>(K), Xdq);
    }
  }
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (T + 7) / 8;
  const int blocks = static_cast<int>(want < 4 * sms ? want : 4 * sms);
  codes_to_xdq_kernel<<<blocks, 256, 0, stream>>>(Xq, s_x, static_cast<int>(T),
                                                  static_cast<int>(K), Xdq);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_act_quant_fp8(const uint16_t* X, int64_t T, int64_t K, uint8_t* Xq8, float* s8,
                         uint16_t* Xdq, cudaStream_t stream) {
  return launch_aq<true>(X, T, K, reinterpret_cast<int8_t*>(Xq8), s8, nullptr, Xdq, stream);
}

int launch_codes_to_fp8(const int8_t* W, int64_t numel, uint8_t* W8, cudaStream_t stream) {
  const int threads = 256;
  codes_to_fp8_kernel<<<grid_for((numel >> 4) + 1, threads), threads, 0, stream>>>(W, numel, W8);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_codes_to_fp8_split(const int8_t* W, int64_t N, int64_t K, uint8_t* W8,
                              cudaStream_t stream) {
  const int threads = 256;
  codes_to_fp8_split_kernel<<<grid_for(N * (K >> 4), threads), threads, 0, stream>>>(W, N, K, W8);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_codes_to_bf16(const int8_t* W, int64_t numel, uint16_t* W_img, cudaStream_t stream) {
  const int threads = 256;
  codes_to_bf16_kernel<<<grid_for((numel >> 6) + 1, threads), threads, 0, stream>>>(W, numel, W_img);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_absmean_partial(const float* W0, int64_t numel, double* ws, cudaStream_t stream) {
  absmean_partial_kernel<<<kAbsmeanBlocks, kAbsThreads, 0, stream>>>(W0, numel, ws);
  absmean_final_kernel<<<1, kAbsmeanBlocks, 0, stream>>>(ws);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

int launch_absmean_codes(const float* W0, int64_t numel, float s_w, int32_t qmin, int32_t qmax,
                         int8_t* codes, cudaStream_t stream) {
  const int threads = 256;
  absmean_codes_kernel<<<grid_for(numel, threads), threads, 0, stream>>>(W0, numel, s_w, qmin,
                                                                         qmax, codes);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

}  // namespace dqt

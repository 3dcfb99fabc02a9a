// The three dense contractions of a DQT BitLinear training step on the GB300
// 5th-generation tensor cores (tcgen05.mma kind::f16, fp32 accumulator in
// tensor memory), operands staged by TMA into 128-byte-swizzled shared memory:
//
//   forward  Y  = X_tilde W_tilde^T   (Sec. 3.2)  exact integer accumulation
//   dX          = dY W_tilde          (Sec. 3.2; no STE on the weight)
//   dW          = dY^T X_tilde        (Sec. 3.2) fused with AdamW (Sec. 4.1) and
//                                     W_hat = SR(W') (Eq. 1, Eq. 5) in the epilogue
//
// One CTA computes one 128 x BN output tile with three warp roles:
//   warp 0     TMA producer (one lane), kStages-deep ring of A/B stages
//   warp 1     tensor-memory allocator and MMA issuer (one lane)
//   warps 2-5  epilogue: tensor memory -> registers -> global memory
//
// Integer exactness of the forward GEMM.  The codes are fed as bf16 values
// (exact for |v| <= 256); each product is exact in fp32 and a sum of integers
// stays exact while its magnitude is at most 2^24.  The reduction is split into
// chunks of chunk_k elements with chunk_k * 128 * max|c| <= 2^24; after each
// chunk but the last the epilogue converts the fp32 partial to int32 and adds
// it to a running int32 sum kept in the second half of the tensor memory.
// Ternary weights (max|c| = 1) need no drain for K <= 131072.
#include <cuda.h>

#include "dqt_internal.h"

namespace dqt {

namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // bf16 per 128-byte swizzled row
constexpr int kStages = 4;
constexpr int kThreads = 192;
constexpr uint64_t kDrainNs = 1000000000ull;  // wait for in-flight copies/MMAs on abort

struct Params {
  int M, N, Kred, num_kb, chunk_kb;
  uint64_t wait_ns;
  unsigned int* status;
  const float* s_x;
  float scale;
  __nv_bfloat16* out_bf16;
  int32_t* acc_out;
  int8_t* W;
  float* m;
  float* v;
  float* dW_out;
  unsigned long long* changed;
  UpdateConsts uc;
};

template <int BN>
struct Smem {
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int BAR_OFF = kStages * STAGE_BYTES;
  static constexpr int BYTES = BAR_OFF + 256 + 1024;  // + barriers + alignment slack
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  const uint32_t s = smem_u32(p);
  return p + ((1024u - (s & 1023u)) & 1023u);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// Warp-uniform bounded wait: every lane waits, the warp fails if any lane did.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t ns) {
  const bool ok = mbar_wait(bar, parity, ns);
  return __all_sync(0xffffffffu, ok);
}

template <int BN, bool A_MN, bool B_MN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const Params p) {
  using S = Smem<BN>;
  constexpr uint32_t IDESC = idesc_bf16(BM, BN, A_MN, B_MN);
  constexpr uint32_t TMEM_COLS = (EPI == GEMM_FWD) ? 2 * BN : BN;
  constexpr uint32_t MN_CHUNK_BYTES = 64 * BK * 2;  // one 64-wide MN box of BK rows

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages * S::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::BAR_OFF);
  uint64_t* empty = full + kStages;
  uint64_t* acc_full = empty + kStages;
  uint64_t* acc_empty = acc_full + 1;
  uint64_t* drain_bar = acc_full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int m0 = blockIdx.x * BM;
  const int n0 = blockIdx.y * BN;
  const int nchunks = (p.num_kb + p.chunk_kb - 1) / p.chunk_kb;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 4);
    mbar_init(drain_bar, 1);
    fence_mbarrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) tmem_alloc(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int issued = 0;
      bool ok = true;
      for (int kb = 0; kb < p.num_kb; ++kb) {
        const int s = kb % kStages;
        const uint32_t ph = (kb / kStages) & 1u;
        if (kb >= kStages && !mbar_wait(&empty[s], ph ^ 1u, p.wait_ns)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&full[s], S::STAGE_BYTES);
        uint8_t* a = sA + s * S::A_BYTES;
        uint8_t* b = sB + s * S::B_BYTES;
        const int k0 = kb * BK;
        if (!A_MN) {
          tma_load_2d(&tmA, &full[s], a, k0, m0);
        } else {
#pragma unroll
          for (int j = 0; j < BM / 64; ++j)
            tma_load_2d(&tmA, &full[s], a + j * MN_CHUNK_BYTES, m0 + 64 * j, k0);
        }
        if (!B_MN) {
          tma_load_2d(&tmB, &full[s], b, k0, n0);
        } else {
#pragma unroll
          for (int j = 0; j < BN / 64; ++j)
            tma_load_2d(&tmB, &full[s], b + j * MN_CHUNK_BYTES, n0 + 64 * j, k0);
        }
        ++issued;
      }
      if (!ok) {
        record_timeout(p.status);
        // Let the (at most kStages) copies still in flight land before exit.
        for (int i = (issued > kStages ? issued - kStages : 0); i < issued; ++i)
          mbar_wait(&full[i % kStages], (i / kStages) & 1u, kDrainNs);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      bool ok = true;
      for (int kb = 0; kb < p.num_kb; ++kb) {
        const int s = kb % kStages;
        const uint32_t ph = (kb / kStages) & 1u;
        const int kc = kb % p.chunk_kb;
        const int chunk = kb / p.chunk_kb;
        if (kc == 0 && chunk > 0) {
          // The epilogue must have drained the previous chunk's partial sums.
          if (!mbar_wait(acc_empty, (chunk - 1) & 1u, p.wait_ns)) {
            ok = false;
            break;
          }
        }
        if (!mbar_wait(&full[s], ph, p.wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_base = smem_u32(sA + s * S::A_BYTES);
        const uint32_t b_base = smem_u32(sB + s * S::B_BYTES);
#pragma unroll
        for (int ks = 0; ks < BK / 16; ++ks) {
          const uint64_t ad = A_MN ? sdesc_sw128(a_base + ks * 2048, MN_CHUNK_BYTES, 1024)
                                   : sdesc_sw128(a_base + ks * 32, 16, 1024);
          const uint64_t bd = B_MN ? sdesc_sw128(b_base + ks * 2048, MN_CHUNK_BYTES, 1024)
                                   : sdesc_sw128(b_base + ks * 32, 16, 1024);
          umma_bf16(tmem, ad, bd, IDESC, (kc > 0 || ks > 0) ? 1u : 0u);
        }
        umma_commit(&empty[s]);
        if (kc == p.chunk_kb - 1 || kb == p.num_kb - 1) umma_commit(acc_full);
      }
      if (!ok) {
        record_timeout(p.status);
        umma_commit(drain_bar);  // every MMA issued so far has finished
        mbar_wait(drain_bar, 0, kDrainNs);
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5) ----------------
    const int quad = warp & 3;  // tensor-memory lanes this warp may access
    const int row = quad * 32 + lane;
    const int gm = m0 + row;
    const bool row_ok = gm < p.M;
    const uint32_t t_row = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    bool ok = true;
    for (int c = 0; c < nchunks && ok; ++c) {
      ok = warp_wait(acc_full, c & 1u, p.wait_ns);
      if (!ok) break;
      tc_fence_after();
      if (c + 1 < nchunks) {
        // Drain an exact fp32 chunk into the int32 running sum (forward only).
#pragma unroll 1
        for (int cc = 0; cc < BN / 32; ++cc) {
          uint32_t a[32], r[32];
          tmem_ld_32x32b_x32(t_row + cc * 32, a);
          if (c > 0) tmem_ld_32x32b_x32(t_row + BN + cc * 32, r);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int32_t part = __float2int_rn(__uint_as_float(a[i]));
            r[i] = static_cast<uint32_t>((c > 0 ? static_cast<int32_t>(r[i]) : 0) + part);
          }
          tmem_st_32x32b_x32(t_row + BN + cc * 32, r);
        }
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acc_empty);
        continue;
      }

      // ---- final chunk: the tile's epilogue ----
      if (EPI == GEMM_FWD) {
        float a_t = 0.0f;
        if (row_ok) a_t = __fdiv_rn(1.0f, __fmul_rn(p.s_x[gm], p.scale));
#pragma unroll 1
        for (int cc = 0; cc < BN / 32; ++cc) {
          uint32_t a[32], r[32];
          tmem_ld_32x32b_x32(t_row + cc * 32, a);
          if (nchunks > 1) tmem_ld_32x32b_x32(t_row + BN + cc * 32, r);
          tmem_ld_wait();
          const int gn0 = n0 + cc * 32;
          if (!row_ok || gn0 >= p.N) continue;
          int32_t acc[32];
#pragma unroll
          for (int i = 0; i < 32; ++i)
            acc[i] = __float2int_rn(__uint_as_float(a[i])) +
                     (nchunks > 1 ? static_cast<int32_t>(r[i]) : 0);
          __nv_bfloat16* yrow = p.out_bf16 + static_cast<size_t>(gm) * p.N + gn0;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            if (gn0 + 8 * j >= p.N) break;
            uint4 pk;
            pk.x = pack_bf16x2(__fmul_rn(__int2float_rn(acc[8 * j + 0]), a_t),
                               __fmul_rn(__int2float_rn(acc[8 * j + 1]), a_t));
            pk.y = pack_bf16x2(__fmul_rn(__int2float_rn(acc[8 * j + 2]), a_t),
                               __fmul_rn(__int2float_rn(acc[8 * j + 3]), a_t));
            pk.z = pack_bf16x2(__fmul_rn(__int2float_rn(acc[8 * j + 4]), a_t),
                               __fmul_rn(__int2float_rn(acc[8 * j + 5]), a_t));
            pk.w = pack_bf16x2(__fmul_rn(__int2float_rn(acc[8 * j + 6]), a_t),
                               __fmul_rn(__int2float_rn(acc[8 * j + 7]), a_t));
            *reinterpret_cast<uint4*>(yrow + 8 * j) = pk;
          }
          if (p.acc_out) {
            int32_t* arow = p.acc_out + static_cast<size_t>(gm) * p.N + gn0;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              if (gn0 + 4 * j >= p.N) break;
              *reinterpret_cast<int4*>(arow + 4 * j) =
                  make_int4(acc[4 * j], acc[4 * j + 1], acc[4 * j + 2], acc[4 * j + 3]);
            }
          }
        }
      } else if (EPI == GEMM_DX) {
#pragma unroll 1
        for (int cc = 0; cc < BN / 32; ++cc) {
          uint32_t a[32];
          tmem_ld_32x32b_x32(t_row + cc * 32, a);
          tmem_ld_wait();
          const int gn0 = n0 + cc * 32;
          if (!row_ok || gn0 >= p.N) continue;
          __nv_bfloat16* yrow = p.out_bf16 + static_cast<size_t>(gm) * p.N + gn0;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            if (gn0 + 8 * j >= p.N) break;
            uint4 pk;
            const float* f = reinterpret_cast<const float*>(a) + 8 * j;
            pk.x = pack_bf16x2(__fmul_rn(f[0], p.scale), __fmul_rn(f[1], p.scale));
            pk.y = pack_bf16x2(__fmul_rn(f[2], p.scale), __fmul_rn(f[3], p.scale));
            pk.z = pack_bf16x2(__fmul_rn(f[4], p.scale), __fmul_rn(f[5], p.scale));
            pk.w = pack_bf16x2(__fmul_rn(f[6], p.scale), __fmul_rn(f[7], p.scale));
            *reinterpret_cast<uint4*>(yrow + 8 * j) = pk;
          }
        }
      } else {  // GEMM_DW: gradient -> AdamW -> SR -> codes, all in registers
        uint32_t n_changed = 0;
#pragma unroll 1
        for (int cc = 0; cc < BN / 32; ++cc) {
          uint32_t a[32];
          tmem_ld_32x32b_x32(t_row + cc * 32, a);
          tmem_ld_wait();
          const int gk0 = n0 + cc * 32;
          if (!row_ok || gk0 >= p.N) continue;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int gk = gk0 + 4 * j;
            if (gk >= p.N) break;
            const size_t e = static_cast<size_t>(gm) * p.N + gk;
            float4 g4 = make_float4(__uint_as_float(a[4 * j]), __uint_as_float(a[4 * j + 1]),
                                    __uint_as_float(a[4 * j + 2]), __uint_as_float(a[4 * j + 3]));
            if (p.dW_out) *reinterpret_cast<float4*>(p.dW_out + e) = g4;
            if (p.W) {
              char4 c4 = *reinterpret_cast<const char4*>(p.W + e);
              float4 m4 = *reinterpret_cast<const float4*>(p.m + e);
              float4 v4 = *reinterpret_cast<const float4*>(p.v + e);
              uint4 w = make_uint4(0, 0, 0, 0);
              if (p.uc.round_mode == 0)
                w = sr_words(e >> 2, p.uc.step_lo, p.uc.tensor_id, p.uc.key0, p.uc.key1);
              const int32_t n0c = dqt_update_elem(p.uc, g4.x, c4.x, m4.x, v4.x, w.x);
              const int32_t n1c = dqt_update_elem(p.uc, g4.y, c4.y, m4.y, v4.y, w.y);
              const int32_t n2c = dqt_update_elem(p.uc, g4.z, c4.z, m4.z, v4.z, w.z);
              const int32_t n3c = dqt_update_elem(p.uc, g4.w, c4.w, m4.w, v4.w, w.w);
              n_changed += (n0c != c4.x) + (n1c != c4.y) + (n2c != c4.z) + (n3c != c4.w);
              *reinterpret_cast<char4*>(p.W + e) = make_char4(static_cast<signed char>(n0c),
                                                              static_cast<signed char>(n1c),
                                                              static_cast<signed char>(n2c),
                                                              static_cast<signed char>(n3c));
              *reinterpret_cast<float4*>(p.m + e) = m4;
              *reinterpret_cast<float4*>(p.v + e) = v4;
            }
          }
        }
        if (p.changed) {
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) n_changed += __shfl_xor_sync(0xffffffffu, n_changed, off);
          if (lane == 0 && n_changed) atomicAdd(p.changed, static_cast<unsigned long long>(n_changed));
        }
      }
    }
    if (!ok && lane == 0) record_timeout(p.status);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// Host side: tensor maps and launch.
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2-D bf16 row-major matrix with `inner` contiguous elements per row and
// `outer` rows; box of box_inner x box_outer, 128-byte swizzle, zero fill.
bool make_map(CUtensorMap* map, const void* ptr, uint64_t inner, uint64_t outer,
              uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {inner * 2};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, bool A_MN, bool B_MN, int EPI>
int launch_tile_kernel(const CUtensorMap& ta, const CUtensorMap& tb, const Params& p,
                       cudaStream_t stream) {
  auto kern = gemm_kernel<BN, A_MN, B_MN, EPI>;
  const int smem = Smem<BN>::BYTES;
  static bool attr_set = false;  // per template instance
  if (!attr_set) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
        cudaSuccess)
      return 3;
    attr_set = true;
  }
  dim3 grid((p.M + BM - 1) / BM, (p.N + BN - 1) / BN);
  kern<<<grid, kThreads, smem, stream>>>(ta, tb, p);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

}  // namespace

int launch_gemm(const GemmLaunch& g, cudaStream_t stream) {
  constexpr int BN = 256;
  Params p{};
  p.M = g.M;
  p.N = g.N;
  p.Kred = g.Kred;
  p.num_kb = (g.Kred + BK - 1) / BK;
  p.chunk_kb = p.num_kb;
  if (g.kind == GEMM_FWD) {
    const int ck = g.chunk_k / BK;
    if (ck < 1) return 1;
    if (ck < p.num_kb) p.chunk_kb = ck;
  }
  p.wait_ns = wait_limit_ns();
  p.status = status_word();
  if (!p.status) return 3;
  p.s_x = g.s_x;
  p.scale = g.scale;
  p.out_bf16 = static_cast<__nv_bfloat16*>(g.out_bf16);
  p.acc_out = g.acc_out;
  p.W = g.W;
  p.m = g.m;
  p.v = g.v;
  p.dW_out = g.dW_out;
  p.changed = g.changed;
  p.uc = g.uc;

  CUtensorMap ta, tb;
  switch (g.kind) {
    case GEMM_FWD:
      if (!make_map(&ta, g.A, g.Kred, g.M, BK, BM)) return 3;
      if (!make_map(&tb, g.B, g.Kred, g.N, BK, BN)) return 3;
      return launch_tile_kernel<BN, false, false, GEMM_FWD>(ta, tb, p, stream);
    case GEMM_DX:
      if (!make_map(&ta, g.A, g.Kred, g.M, BK, BM)) return 3;
      if (!make_map(&tb, g.B, g.N, g.Kred, 64, BK)) return 3;
      return launch_tile_kernel<BN, false, true, GEMM_DX>(ta, tb, p, stream);
    case GEMM_DW:
      if (!make_map(&ta, g.A, g.M, g.Kred, 64, BK)) return 3;
      if (!make_map(&tb, g.B, g.N, g.Kred, 64, BK)) return 3;
      return launch_tile_kernel<BN, true, true, GEMM_DW>(ta, tb, p, stream);
  }
  return 1;
}

}  // namespace dqt

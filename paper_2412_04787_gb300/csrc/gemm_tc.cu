// The three dense contractions of a DQT BitLinear training step on the GB300
// 5th-generation tensor cores (tcgen05.mma kind::f16, fp32 accumulator in
// tensor memory), operands staged by TMA into 128-byte-swizzled shared memory:
//
//   forward  Y  = X_tilde W_tilde^T   (Sec. 3.2)  exact integer accumulation
//   dX          = dY W_tilde          (Sec. 3.2; no STE on the weight)
//   dW          = dY^T X_tilde        (Sec. 3.2) fused with AdamW (Sec. 4.1) and
//                                     W_hat = SR(W') (Eq. 1, Eq. 5) in the epilogue
//
// Two persistent kernels walk output tiles in a static round-robin order:
//
//   gemm_pair_kernel (default): a cluster of two CTAs on one TPC computes a
//     256 x 256 tile with tcgen05.mma.cta_group::2; each CTA stages its 128
//     rows of A and its half of B, and the leader's single MMA-issuing lane
//     drives both SMs' tensor cores.
//   gemm_kernel (dqt_set_gemm_tiles(1)): one CTA per SM, 128 x 256 tiles.
//
// Warp roles (both kernels):
//   warp 0     TMA producer (one lane): a ring of A/B stages that runs
//              continuously across tiles
//   warp 1     tensor-memory allocator and MMA issuer (one lane)
//   warps 2+   epilogue: tensor memory -> registers -> global memory; each
//              tensor-memory lane quadrant is served by the same number of
//              warps (8 epilogue warps, 16 for the dW update and the drained
//              8-bit forward of the 2-SM kernel)
// The accumulator is double-buffered in tensor memory, so the epilogue of one
// tile (for dW: the whole AdamW + stochastic-rounding update) overlaps the
// MMAs of the next.
//
// FP8 environment (Sec. 4.1/4.3): the forward also runs on E4M3 operands
// (tcgen05.mma kind::f8f6f4, 2-SM tiles only): a 128-byte swizzled row then
// holds 128 elements of K, so a stage carries twice the reduction of a bf16
// stage in the same bytes, and Y = bf16(acc * 1/(s_x s_w)) from the fp32
// accumulator.
//
// Integer exactness of the forward GEMM.  The codes are fed as bf16 values
// (exact for |v| <= 256); each product is exact in fp32 and a sum of integers
// stays exact while its magnitude is at most 2^24.  The reduction is split into
// chunks of chunk_k elements with chunk_k * 128 * max|c| <= 2^24.  With more
// than one chunk (8-bit codes, K > 1024) every chunk is its own accumulation
// unit; the epilogue converts each chunk's exact fp32 sum to int32 and adds it
// to running sums: in registers (the 2-SM kernel, 16 epilogue warps) or in a
// third tensor-memory region (the 1-SM kernel, BN = 128).  Ternary weights
// (max|c| = 1) need no drain for K <= 131072.
#include <cuda.h>
#include <cuda_fp8.h>

#include <atomic>

#include "dqt_internal.h"

namespace dqt {

static_assert(sizeof(UpdateConsts) <= 80, "update constants fit the shared barrier area");

namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // bf16 per 128-byte swizzled row
constexpr int kStages = 4;
constexpr int kEpiWarps = 8;
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr uint64_t kDrainNs = 1000000000ull;  // wait for in-flight copies/MMAs on abort

// Philox4x32-10 (the generator of sr_words) for the elements of one update
// call: the round keys and, in the first round, the product of counter word
// 2 (the step) and word 3 (the weight tensor) are the same for every
// element, so the host computes them once (philox_call_consts).
struct PhiloxCall {
  uint32_t rk[20];  // rk[2r], rk[2r + 1]: round r's keys, key0 + r W0 and key1 + r W1
  uint32_t c0x;     // hi(M1 * step) ^ rk[0]: round 0's first output word before ^ counter word 1
  uint32_t c0y;     // lo(M1 * step): round 0's second output word
  uint32_t x3k;     // tensor id ^ rk[1]
};

struct Params {
  int M, N, Kred, num_kb, chunk_kb;
  int num_n, num_tiles;
  uint64_t wait_ns;
  unsigned int* status;
  const float* s_x;
  float scale;
  __nv_bfloat16* out_bf16;
  int32_t* acc_out;
  float* acc_f32;  // FP8 forward: optional fp32 accumulators
  int8_t* W;
  bool packed;  // W holds 2-bit packed ternary codes (one byte per 4 weights)
  float* m;
  float* v;
  float* dW_out;
  unsigned long long* changed;
  UpdateConsts uc;
  const UpdateConsts* uc_dev;  // if set, the update constants are read from here at run time
  // split-T (2-SM dW only): work unit t covers tile t / splits and the token
  // slice of k-blocks [s * kb_per_split, ...), s = t % splits; its fp32
  // partial goes to dW_out + s * slab
  int splits, kb_per_split;
  long long slab;
  // tail (2-SM dW with splits == 1): units below full_units are whole tiles
  // with the fused epilogue; the tiles from full_tiles on are each cut into
  // tail_splits token slices of tail_kbps k-blocks, one unit each, whose fp32
  // partials go to `part` (slice s of tail tile j at (s * tail_tiles + j) *
  // 65536 floats, tile-local row-major 256 x 256) for a streaming kernel that
  // sums them in slice order and applies the update.
  int full_units, full_tiles, tail_tiles, tail_splits, tail_kbps;
  float* part;
  // forward / dX tail: the slices of a tile region are added by the last of
  // them to finish, found with one counter per (tail tile, CTA rank,
  // epilogue warp): (tag << 16) | slices done, tag unique per launch, so a
  // counter left by an earlier launch counts as zero
  unsigned long long* tail_ctr;
  unsigned long long tail_tag;
  // two weights stacked in one call (e.g. a LLaMA MLP's gate and up
  // projections, which read the same input): output columns (forward) or
  // output rows (dW) from `split` on, a multiple of 256 (whole tiles), belong
  // to the second weight, with its own scale (scale1) and update constants
  // (uc1), and its Philox elements counted from its own first element; 0: one
  // weight
  int split;
  float scale1;
  UpdateConsts uc1;
  // 2-SM kernels: output tiles numbered down the columns (tile % num_m is
  // the row tile) instead of along the rows: the A operand is then the one
  // every wave re-reads (chosen when A's panels are the smaller set)
  int num_m;
  bool col_major;
  // dW: if set, the bf16 image of every updated code is written here too
  // (the next forward's operand), at the code's element index
  __nv_bfloat16* img_next;
  // dW: if set, the E4M3 image of every updated code (the next FP8 forward's
  // operand; exact for |code| <= 16), or with img8_split the split image
  // [M, 2N] of wider codes: 16 (c >> 4) at column gk of row gm, c & 15 at N + gk
  uint8_t* img8_next;
  int img8_split;
  // dW with the constants in the parameter space: the parts of the
  // stochastic-rounding generator that are the same for every element of
  // the call, for uc and uc1
  PhiloxCall pc, pc1;
  // FWD8 on split codes: A's k-block kb is read from column (kb * 128) mod
  // a_wrap (the activation row serves both halves of the split weight row)
  int a_wrap;
};

// The bf16 image of four codes (exact: integers of magnitude <= 128).
__device__ __forceinline__ void store_code_image4(__nv_bfloat16* img, size_t e, int32_t a, int32_t b,
                                                  int32_t c, int32_t d);

// The E4M3 image of four codes (exact for |code| <= 16).
__device__ __forceinline__ void store_code_e4m3_4(uint8_t* img8, size_t e, int32_t a, int32_t b,
                                                  int32_t c, int32_t d);

// The E4M3 image of four updated codes at element e = gm N + gk, direct or split.
__device__ __forceinline__ void store_img8(const Params& p, size_t e, int gm, int32_t a, int32_t b,
                                           int32_t c, int32_t d);

// Row and column tile (256 x 256) of a 2-SM kernel's tile index.
__device__ __forceinline__ int pair_tile_m(const Params& p, int tile) {
  return p.col_major ? tile % p.num_m : tile / p.num_n;
}
__device__ __forceinline__ int pair_tile_n(const Params& p, int tile) {
  return p.col_major ? tile / p.num_m : tile % p.num_n;
}

struct Unit {
  int tile, kb0, kb1;
  int slab;   // split-T slab of the unit's partial (0 without split-T)
  int slice;  // tail slice, -1 for a whole tile
};

__device__ __forceinline__ Unit decode_unit(const Params& p, int t) {
  Unit u;
  if (t < p.full_units) {
    u.tile = t / p.splits;
    u.slab = t - u.tile * p.splits;
    u.kb0 = u.slab * p.kb_per_split;
    u.kb1 = min(p.num_kb, u.kb0 + p.kb_per_split);
    u.slice = -1;
  } else {
    const int q = t - p.full_units;
    const int j = q / p.tail_splits;
    u.tile = p.full_tiles + j;
    u.slice = q - j * p.tail_splits;
    u.slab = 0;
    u.kb0 = u.slice * p.tail_kbps;
    u.kb1 = min(p.num_kb, u.kb0 + p.tail_kbps);
  }
  return u;
}

constexpr int kStageLd = 33;  // padded row pitch (floats) of the epilogue transpose buffer

template <int BN, int EPI>
struct Smem {
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  // dW: one 32 x 33 fp32 transpose buffer per epilogue warp
  static constexpr int XPOSE_OFF = kStages * STAGE_BYTES;
  static constexpr int XPOSE_BYTES = (EPI == GEMM_DW) ? kEpiWarps * 32 * kStageLd * 4 : 0;
  static constexpr int BAR_OFF = XPOSE_OFF + XPOSE_BYTES;
  static constexpr int BYTES = BAR_OFF + 256 + 1024;  // + barriers + alignment slack
  static_assert(BYTES <= 232448, "shared memory per CTA");
  static_assert((2 * kStages + 5) * 8 + 4 <= 128, "barrier area: barriers, then the update constants");
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  const uint32_t s = smem_u32(p);
  return p + ((1024u - (s & 1023u)) & 1023u);
}

// Invalidate the 128-byte L2 line at p (128-byte aligned) without writing it
// back: for data that is dead once read (slice partials).
__device__ __forceinline__ void l2_discard_line(const void* p) {
  asm volatile("discard.global.L2 [%0], 128;" ::"l"(p) : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ void store_code_e4m3_4(uint8_t* img8, size_t e, int32_t a, int32_t b,
                                                  int32_t c, int32_t d) {
  const uint32_t lo = __nv_cvt_float2_to_fp8x2(make_float2(static_cast<float>(a), static_cast<float>(b)),
                                               __NV_SATFINITE, __NV_E4M3);
  const uint32_t hi = __nv_cvt_float2_to_fp8x2(make_float2(static_cast<float>(c), static_cast<float>(d)),
                                               __NV_SATFINITE, __NV_E4M3);
  __stcs(reinterpret_cast<uint32_t*>(img8 + e), (lo & 0xFFFFu) | ((hi & 0xFFFFu) << 16));
}

__device__ __forceinline__ void store_img8(const Params& p, size_t e, int gm, int32_t a, int32_t b,
                                           int32_t c, int32_t d) {
  if (!p.img8_split) {
    store_code_e4m3_4(p.img8_next, e, a, b, c, d);
    return;
  }
  // split row gm of 2N bytes: the high halves at gm 2N + gk = e + gm N, the low N later
  const size_t h = e + static_cast<size_t>(gm) * p.N;
  store_code_e4m3_4(p.img8_next, h, 16 * (a >> 4), 16 * (b >> 4), 16 * (c >> 4), 16 * (d >> 4));
  store_code_e4m3_4(p.img8_next, h + p.N, a & 15, b & 15, c & 15, d & 15);
}

__device__ __forceinline__ void store_code_image4(__nv_bfloat16* img, size_t e, int32_t a, int32_t b,
                                                  int32_t c, int32_t d) {
  __stcs(reinterpret_cast<uint2*>(img + e),
         make_uint2(pack_bf16x2(static_cast<float>(a), static_cast<float>(b)),
                    pack_bf16x2(static_cast<float>(c), static_cast<float>(d))));
}

// Warp-uniform bounded wait: every lane waits, the warp fails if any lane did.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t ns) {
  const bool ok = mbar_wait(bar, parity, ns);
  return __all_sync(0xffffffffu, ok);
}

// ---------------------------------------------------------------------------
// Epilogues.  Each processes 32 consecutive columns [gn0, gn0 + 32) of one
// output row gm, given the fp32 accumulator values a[] (and, for the forward
// GEMM with drained chunks, the running int32 sums r[]).
// ---------------------------------------------------------------------------
__device__ __forceinline__ void epi_fwd(const Params& p, int gm, int gn0, float a_t,
                                        const uint32_t (&a)[32], const uint32_t (&r)[32],
                                        bool add_running) {
  int32_t acc[32];
#pragma unroll
  for (int i = 0; i < 32; ++i)
    acc[i] = __float2int_rn(__uint_as_float(a[i])) + (add_running ? static_cast<int32_t>(r[i]) : 0);
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

// The forward's output from exact int32 accumulators (drained chunks).
__device__ __forceinline__ void epi_fwd_int(const Params& p, int gm, int gn0, float a_t,
                                            const int32_t (&acc)[32]) {
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

__device__ __forceinline__ void epi_dx(const Params& p, int gm, int gn0, const uint32_t (&a)[32]) {
  __nv_bfloat16* yrow = p.out_bf16 + static_cast<size_t>(gm) * p.N + gn0;
  const float* f = reinterpret_cast<const float*>(a);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (gn0 + 8 * j >= p.N) break;
    uint4 pk;
    pk.x = pack_bf16x2(__fmul_rn(f[8 * j + 0], p.scale), __fmul_rn(f[8 * j + 1], p.scale));
    pk.y = pack_bf16x2(__fmul_rn(f[8 * j + 2], p.scale), __fmul_rn(f[8 * j + 3], p.scale));
    pk.z = pack_bf16x2(__fmul_rn(f[8 * j + 4], p.scale), __fmul_rn(f[8 * j + 5], p.scale));
    pk.w = pack_bf16x2(__fmul_rn(f[8 * j + 6], p.scale), __fmul_rn(f[8 * j + 7], p.scale));
    *reinterpret_cast<uint4*>(yrow + 8 * j) = pk;
  }
}

// FP8 forward: the fp32 accumulators are not integers; Y = bf16(acc * a_t).
__device__ __forceinline__ void epi_fwd8(const Params& p, int gm, int gn0, float a_t,
                                         const uint32_t (&a)[32]) {
  const float* f = reinterpret_cast<const float*>(a);
  __nv_bfloat16* yrow = p.out_bf16 + static_cast<size_t>(gm) * p.N + gn0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (gn0 + 8 * j >= p.N) break;
    uint4 pk;
    pk.x = pack_bf16x2(__fmul_rn(f[8 * j + 0], a_t), __fmul_rn(f[8 * j + 1], a_t));
    pk.y = pack_bf16x2(__fmul_rn(f[8 * j + 2], a_t), __fmul_rn(f[8 * j + 3], a_t));
    pk.z = pack_bf16x2(__fmul_rn(f[8 * j + 4], a_t), __fmul_rn(f[8 * j + 5], a_t));
    pk.w = pack_bf16x2(__fmul_rn(f[8 * j + 6], a_t), __fmul_rn(f[8 * j + 7], a_t));
    *reinterpret_cast<uint4*>(yrow + 8 * j) = pk;
  }
  if (p.acc_f32) {
    float* arow = p.acc_f32 + static_cast<size_t>(gm) * p.N + gn0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (gn0 + 4 * j >= p.N) break;
      *reinterpret_cast<float4*>(arow + 4 * j) =
          make_float4(f[4 * j], f[4 * j + 1], f[4 * j + 2], f[4 * j + 3]);
    }
  }
}

// dW: gradient -> AdamW -> SR -> codes, in registers, four weights (one
// Philox block) per lane at a time.  A warp owns 32 rows (its tensor-memory
// lanes) and a run of 32-column chunks of the tile.  Each chunk's 32 x 32
// gradient block is transposed through a padded shared buffer so that eight
// lanes share a row: every optimiser-state access of the warp covers four
// full 128-byte row segments instead of 32 scattered ones.  The loads are
// software-pipelined in half-chunks (four rows per lane): the next half's
// codes, m and v are in flight while the current half is updated.  Streaming
// cache hints keep the optimiser state from evicting GEMM operands from L2.
struct DwLoads {
  float4 m[4], v[4];
  char4 c[4];
};

template <bool PK>
__device__ __forceinline__ void dw_issue(const Params& p, int row0, int gn0, int h, int lane,
                                         DwLoads& L) {
  const int gk = gn0 + (lane & 7) * 4;
  if (!p.W || gn0 >= p.N || gk >= p.N) return;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int gm = row0 + (lane >> 3) + 4 * (4 * h + j);
    if (gm < p.M) {
      const size_t e = static_cast<size_t>(gm) * p.N + gk;
      L.c[j] = PK ? tern_unpack4(__ldcs(reinterpret_cast<const uint8_t*>(p.W) + (e >> 2)))
                  : __ldcs(reinterpret_cast<const char4*>(p.W + e));
      L.m[j] = __ldcs(reinterpret_cast<const float4*>(p.m + e));
      L.v[j] = __ldcs(reinterpret_cast<const float4*>(p.v + e));
    }
  }
}

template <bool PK>
__device__ __forceinline__ uint32_t dw_update(const Params& p, const UpdateConsts& uc, size_t e_off,
                                              float* dw_out, int row0, int gn0, int h, int lane,
                                              const float* xp, DwLoads& L) {
  const int cq = (lane & 7) * 4;
  const int gk = gn0 + cq;
  if (gn0 >= p.N || gk >= p.N) return 0;
  uint32_t n_changed = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int r = (lane >> 3) + 4 * (4 * h + j);
    const int gm = row0 + r;
    if (gm >= p.M) continue;
    const size_t e = static_cast<size_t>(gm) * p.N + gk;
    const float* src = xp + r * kStageLd + cq;
    const float4 g4 = make_float4(src[0], src[1], src[2], src[3]);
    if (dw_out) __stcs(reinterpret_cast<float4*>(dw_out + e), g4);
    if (!p.W) continue;
    uint4 w = make_uint4(0, 0, 0, 0);
    if (uc.round_mode == 0)
      w = sr_words(global_blk(uc, (e - e_off) >> 2), uc.step_lo, uc.tensor_id, uc.key0, uc.key1);
    const int32_t n0c = dqt_update_elem(uc, g4.x, L.c[j].x, L.m[j].x, L.v[j].x, w.x);
    const int32_t n1c = dqt_update_elem(uc, g4.y, L.c[j].y, L.m[j].y, L.v[j].y, w.y);
    const int32_t n2c = dqt_update_elem(uc, g4.z, L.c[j].z, L.m[j].z, L.v[j].z, w.z);
    const int32_t n3c = dqt_update_elem(uc, g4.w, L.c[j].w, L.m[j].w, L.v[j].w, w.w);
    n_changed += (n0c != L.c[j].x) + (n1c != L.c[j].y) + (n2c != L.c[j].z) + (n3c != L.c[j].w);
    if (PK)
      __stcs(reinterpret_cast<uint8_t*>(p.W) + (e >> 2),
             static_cast<uint8_t>(tern_pack4(n0c, n1c, n2c, n3c)));
    else
      __stcs(reinterpret_cast<char4*>(p.W + e),
             make_char4(static_cast<signed char>(n0c), static_cast<signed char>(n1c),
                        static_cast<signed char>(n2c), static_cast<signed char>(n3c)));
    if (p.img_next) store_code_image4(p.img_next, e, n0c, n1c, n2c, n3c);
    if (p.img8_next) store_img8(p, e, gm, n0c, n1c, n2c, n3c);
    __stcs(reinterpret_cast<float4*>(p.m + e), L.m[j]);
    __stcs(reinterpret_cast<float4*>(p.v + e), L.v[j]);
  }
  return n_changed;
}

// Optimiser state of one lane for one row of a half-chunk (4 weights): the
// moments and the codes as loaded (four int8 codes, or one byte of 2-bit
// packed codes, unpacked where they are used).
struct DwRow {
  float4 m, v;
  uint32_t c;
};

__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// The four Philox words of block `blk` (elements 4 blk .. 4 blk + 3), equal
// to sr_words(blk, step, tensor id, key0, key1) of the call's constants.
__device__ __forceinline__ uint4 philox_call(uint64_t blk, const PhiloxCall& k) {
  const uint32_t x0 = static_cast<uint32_t>(blk), x1 = static_cast<uint32_t>(blk >> 32);
  const uint64_t p0 = static_cast<uint64_t>(0xD2511F53u) * x0;
  uint4 c = make_uint4(k.c0x ^ x1, k.c0y, static_cast<uint32_t>(p0 >> 32) ^ k.x3k,
                       static_cast<uint32_t>(p0));
#pragma unroll
  for (int r = 1; r < 10; ++r) {
    const uint64_t q0 = static_cast<uint64_t>(0xD2511F53u) * c.x;
    const uint64_t q1 = static_cast<uint64_t>(0xCD9E8D57u) * c.z;
    c = make_uint4(static_cast<uint32_t>(q1 >> 32) ^ c.y ^ k.rk[2 * r], static_cast<uint32_t>(q1),
                   static_cast<uint32_t>(q0 >> 32) ^ c.w ^ k.rk[2 * r + 1], static_cast<uint32_t>(q0));
  }
  return c;
}

template <bool PK>
__device__ __forceinline__ void dw_load_row(const Params& p, int gm, int gk, DwRow& L) {
  if (!p.W || gk >= p.N || gm >= p.M) return;
  const size_t e = static_cast<size_t>(gm) * p.N + gk;
  L.c = PK ? static_cast<uint32_t>(__ldcs(reinterpret_cast<const uint8_t*>(p.W) + (e >> 2)))
           : __ldcs(reinterpret_cast<const unsigned int*>(p.W + e));
  L.m = __ldcs(reinterpret_cast<const float4*>(p.m + e));
  L.v = __ldcs(reinterpret_cast<const float4*>(p.v + e));
}

template <bool PK, bool FAST>
__device__ __forceinline__ uint32_t dw_update_row(const Params& p, const UpdateConsts& uc,
                                                  const PhiloxCall& pc, size_t e_off,
                                                  float* dw_out, int gm, int gk,
                                                  const float* src, DwRow& L) {
  if (gk >= p.N || gm >= p.M) return 0;
  const size_t e = static_cast<size_t>(gm) * p.N + gk;
  const float4 g4 = make_float4(src[0], src[1], src[2], src[3]);
  if (dw_out) __stcs(reinterpret_cast<float4*>(dw_out + e), g4);
  if (!p.W) return 0;
  const char4 c = PK ? tern_unpack4(L.c)
                     : make_char4(static_cast<signed char>(L.c & 0xFFu),
                                  static_cast<signed char>((L.c >> 8) & 0xFFu),
                                  static_cast<signed char>((L.c >> 16) & 0xFFu),
                                  static_cast<signed char>(L.c >> 24));
  uint4 w = make_uint4(0, 0, 0, 0);
  if (uc.round_mode == 0)
    w = FAST ? philox_call(global_blk(uc, (e - e_off) >> 2), pc)
             : sr_words(global_blk(uc, (e - e_off) >> 2), uc.step_lo, uc.tensor_id, uc.key0, uc.key1);
  const int32_t n0c = dqt_update_elem(uc, g4.x, c.x, L.m.x, L.v.x, w.x);
  const int32_t n1c = dqt_update_elem(uc, g4.y, c.y, L.m.y, L.v.y, w.y);
  const int32_t n2c = dqt_update_elem(uc, g4.z, c.z, L.m.z, L.v.z, w.z);
  const int32_t n3c = dqt_update_elem(uc, g4.w, c.w, L.m.w, L.v.w, w.w);
  if (PK)
    __stcs(reinterpret_cast<uint8_t*>(p.W) + (e >> 2),
           static_cast<uint8_t>(tern_pack4(n0c, n1c, n2c, n3c)));
  else
    __stcs(reinterpret_cast<char4*>(p.W + e),
           make_char4(static_cast<signed char>(n0c), static_cast<signed char>(n1c),
                      static_cast<signed char>(n2c), static_cast<signed char>(n3c)));
  if (p.img_next) store_code_image4(p.img_next, e, n0c, n1c, n2c, n3c);
  if (p.img8_next) store_img8(p, e, gm, n0c, n1c, n2c, n3c);
  __stcs(reinterpret_cast<float4*>(p.m + e), L.m);
  __stcs(reinterpret_cast<float4*>(p.v + e), L.v);
  return (n0c != c.x) + (n1c != c.y) + (n2c != c.z) + (n3c != c.w);
}

// The first half-chunk's state loads of a tile (rows row0 + (lane >> 3) +
// 4 j, columns nbase + 4 (lane & 7) .. + 3).
template <bool PK>
__device__ __forceinline__ void dw_load_first(const Params& p, int row0, int nbase, int lane,
                                              DwRow (&L)[4]) {
#pragma unroll
  for (int j = 0; j < 4; ++j) dw_load_row<PK>(p, row0 + (lane >> 3) + 4 * j, nbase + (lane & 7) * 4, L[j]);
}

// The dW epilogue of one warp for one tile, with the optimiser state loads
// rotated through the registers that hold them: as soon as row j of a
// half-chunk is updated, the loads of row j of the next half-chunk (this
// tile's, or the first of the tile at row0n, nbasen when row0n >= 0) go into
// the same registers, so each load has most of a half-chunk's update to
// arrive in.  On entry L holds the tile's first half-chunk.  Half-chunk q
// covers chunk q / 2 (32 columns at nbase + 32 (q / 2)), rows
// (lane >> 3) + 4 (4 (q % 2) + j), j = 0..3, and columns 4 (lane & 7) .. + 3.
template <bool PK, bool FAST>
__device__ __forceinline__ uint32_t epi_dw_tile_roll(const Params& p, const UpdateConsts& uc,
                                                     const PhiloxCall& pc, size_t e_off,
                                                     float* dw_out, int row0, int nbase,
                                                     int nchunk, uint32_t t_acc, float* xp,
                                                     int lane, DwRow (&L)[4], int row0n,
                                                     int nbasen) {
  const int cq = (lane & 7) * 4;
  const int nq = 2 * nchunk;
  uint32_t n_changed = 0;
#pragma unroll 1
  for (int q = 0; q < nq; ++q) {
    const int h = q & 1;
    const int gn0 = nbase + (q >> 1) * 32;
    if (h == 0) {
      uint32_t a[32];
      tmem_ld_32x32b_x32(t_acc + (q >> 1) * 32, a);
      tmem_ld_wait();
#pragma unroll
      for (int i = 0; i < 32; ++i) xp[lane * kStageLd + i] = __uint_as_float(a[i]);
      __syncwarp();
    }
    const bool in_tile = q + 1 < nq;
    const int nrow0 = in_tile ? row0 : row0n;
    const int ngk = (in_tile ? nbase + ((q + 1) >> 1) * 32 : nbasen) + cq;
    const int nh = in_tile ? (q + 1) & 1 : 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int r = (lane >> 3) + 4 * (4 * h + j);
      n_changed += dw_update_row<PK, FAST>(p, uc, pc, e_off, dw_out, row0 + r, gn0 + cq,
                                           xp + r * kStageLd + cq, L[j]);
      if (nrow0 >= 0) dw_load_row<PK>(p, nrow0 + (lane >> 3) + 4 * (4 * nh + j), ngk, L[j]);
    }
    if (h == 1) __syncwarp();  // the transpose buffer is rewritten for the next chunk
  }
  return n_changed;
}

// The whole dW epilogue of one warp for one tile: `nchunk` chunks of 32
// columns starting at column nbase, rows row0 .. row0 + 31, gradient in
// tensor memory at t_acc (this warp's lanes, chunk cc at column 32 cc).
// With PIPE the next half-chunk's loads are in flight while the current one
// is updated (more registers, for kernels with few epilogue warps).  PK: the
// codes are 2-bit packed ternary (one byte per lane and row).
template <bool PIPE, bool PK>
__device__ __forceinline__ uint32_t epi_dw_tile(const Params& p, const UpdateConsts& uc,
                                                size_t e_off, float* dw_out, int row0, int nbase,
                                                int nchunk, uint32_t t_acc, float* xp, int lane) {
  uint32_t n_changed = 0;
  DwLoads A, B;
  if (PIPE) dw_issue<PK>(p, row0, nbase, 0, lane, A);
#pragma unroll 1
  for (int cc = 0; cc < nchunk; ++cc) {
    const int gn0 = nbase + cc * 32;
    uint32_t a[32];
    tmem_ld_32x32b_x32(t_acc + cc * 32, a);
    tmem_ld_wait();
#pragma unroll
    for (int i = 0; i < 32; ++i) xp[lane * kStageLd + i] = __uint_as_float(a[i]);
    __syncwarp();
    if (PIPE) {
      dw_issue<PK>(p, row0, gn0, 1, lane, B);
      n_changed += dw_update<PK>(p, uc, e_off, dw_out, row0, gn0, 0, lane, xp, A);
      if (cc + 1 < nchunk) dw_issue<PK>(p, row0, gn0 + 32, 0, lane, A);
      n_changed += dw_update<PK>(p, uc, e_off, dw_out, row0, gn0, 1, lane, xp, B);
    } else {
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        dw_issue<PK>(p, row0, gn0, h, lane, A);
        n_changed += dw_update<PK>(p, uc, e_off, dw_out, row0, gn0, h, lane, xp, A);
      }
    }
    __syncwarp();  // the transpose buffer is rewritten for the next chunk
  }
  return n_changed;
}

template <int BN, bool A_MN, bool B_MN, int EPI, bool DRAIN>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const Params p) {
  using S = Smem<BN, EPI>;
  constexpr uint32_t IDESC = idesc_bf16(BM, BN, A_MN, B_MN);
  constexpr uint32_t TMEM_COLS = 512;  // 2 x 256 accumulators, or 3 x 128 with DRAIN
  static_assert(DRAIN ? 3 * BN <= 512 : 2 * BN <= 512, "tensor memory layout");
  constexpr uint32_t RUN_COL = 2 * BN;           // running int32 sums (DRAIN only)
  constexpr uint32_t MN_CHUNK_BYTES = 64 * BK * 2;  // one 64-wide MN box of BK rows
  constexpr int HALF = BN / 2;                   // columns per epilogue warp

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages * S::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::BAR_OFF);
  uint64_t* empty = full + kStages;
  uint64_t* acc_full = empty + kStages;  // [2]
  uint64_t* acc_empty = acc_full + 2;    // [2]
  uint64_t* drain_bar = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  // update constants, read by the dW epilogue from shared memory
  UpdateConsts* uc_s = reinterpret_cast<UpdateConsts*>(smem + S::BAR_OFF + 128);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nchunks = (p.num_kb + p.chunk_kb - 1) / p.chunk_kb;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], kEpiWarps);
    }
    mbar_init(drain_bar, 1);
    if (EPI == GEMM_DW) *uc_s = p.uc_dev ? *p.uc_dev : p.uc;
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
      int it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < p.num_tiles && ok; t += gridDim.x) {
        const int m0 = (t / p.num_n) * BM;
        const int n0 = (t % p.num_n) * BN;
        for (int kb = 0; kb < p.num_kb; ++kb, ++it) {
          const int s = it % kStages;
          const uint32_t ph = (it / kStages) & 1u;
          if (it >= kStages && !mbar_wait(&empty[s], ph ^ 1u, p.wait_ns)) {
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
        }
      }
      if (!ok) record_timeout(p.status);
      // Whatever any role did, the (at most kStages) copies still in flight
      // must land before the CTA exits; in a normal run these are consumed
      // already and each wait returns at once.
      for (int i = (it > kStages ? it - kStages : 0); i < it; ++i)
        mbar_wait(&full[i % kStages], (i / kStages) & 1u, kDrainNs);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      // (short per-k-block loop, as in the 2-SM kernel: incremental stage and
      // phase, descriptors from their precomputed 32-bit halves)
      int s = 0;
      uint32_t ph = 0;
      int u = 0;  // accumulation units (tile chunks) issued so far
      bool ok = true;
      const uint64_t a_desc0 = A_MN ? sdesc_sw128(smem_u32(sA), MN_CHUNK_BYTES, 1024)
                                    : sdesc_sw128(smem_u32(sA), 16, 1024);
      const uint64_t b_desc0 = B_MN ? sdesc_sw128(smem_u32(sB), MN_CHUNK_BYTES, 1024)
                                    : sdesc_sw128(smem_u32(sB), 16, 1024);
      const uint32_t a_lo0 = static_cast<uint32_t>(a_desc0), b_lo0 = static_cast<uint32_t>(b_desc0);
      const uint64_t a_hi = a_desc0 & 0xFFFFFFFF00000000ull, b_hi = b_desc0 & 0xFFFFFFFF00000000ull;
      constexpr uint32_t kAStage = S::A_BYTES >> 4, kBStage = S::B_BYTES >> 4;
      constexpr uint32_t kAStep = A_MN ? (2048 >> 4) : (32 >> 4);
      constexpr uint32_t kBStep = B_MN ? (2048 >> 4) : (32 >> 4);
      for (int t = blockIdx.x; t < p.num_tiles && ok; t += gridDim.x) {
        int kc = 0;  // k-blocks into the current chunk
        for (int kb = 0; kb < p.num_kb; ++kb) {
          const int b = u & 1;
          if (kc == 0 && u >= 2) {
            // The epilogue must have released this accumulator buffer.
            if (!mbar_wait(&acc_empty[b], ((u >> 1) - 1) & 1u, p.wait_ns)) {
              ok = false;
              break;
            }
            tc_fence_after();
          }
          if (!mbar_wait(&full[s], ph, p.wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t alo = a_lo0 + static_cast<uint32_t>(s) * kAStage;
          const uint32_t blo = b_lo0 + static_cast<uint32_t>(s) * kBStage;
          const uint32_t d = tmem + static_cast<uint32_t>(b * BN);
#pragma unroll
          for (int ks = 0; ks < BK / 16; ++ks)
            umma_bf16(d, a_hi | (alo + ks * kAStep), b_hi | (blo + ks * kBStep), IDESC,
                      (kc > 0 || ks > 0) ? 1u : 0u);
          umma_commit(&empty[s]);
          if (++s == kStages) {
            s = 0;
            ph ^= 1u;
          }
          if (++kc == p.chunk_kb || kb == p.num_kb - 1) {
            umma_commit(&acc_full[b]);
            ++u;
            kc = 0;
          }
        }
      }
      if (!ok) record_timeout(p.status);
      // Every MMA issued so far must finish before tensor memory is freed,
      // also when another role gave up first.
      umma_commit(drain_bar);
      mbar_wait(drain_bar, 0, kDrainNs);
    }
  } else {
    // ---------------- epilogue (warps 2..9) ----------------
    const int quad = warp & 3;               // tensor-memory lanes this warp may access
    const int half = (warp - 2) >> 2;        // which half of the tile's columns
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    float* xp = reinterpret_cast<float*>(smem + S::XPOSE_OFF) + (warp - 2) * 32 * kStageLd;
    const UpdateConsts& uc = *uc_s;
    uint32_t n_changed = 0;
    int u = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < p.num_tiles && ok; t += gridDim.x) {
      const int gm = (t / p.num_n) * BM + row;
      const int nbase = (t % p.num_n) * BN + half * HALF;
      const bool row_ok = gm < p.M;
      float a_t = 0.0f;
      if (EPI == GEMM_FWD && row_ok) {
        // the second of two stacked weights (whole tiles of columns): its scale
        const float sw = p.split > 0 && (t % p.num_n) * BN >= p.split ? p.scale1 : p.scale;
        a_t = __fdiv_rn(1.0f, __fmul_rn(p.s_x[gm], sw));
      }
      for (int c = 0; c < nchunks; ++c, ++u) {
        const int b = u & 1;
        ok = warp_wait(&acc_full[b], (u >> 1) & 1u, p.wait_ns);
        if (!ok) break;
        tc_fence_after();
        const uint32_t t_acc = tmem + lane_off + static_cast<uint32_t>(b * BN + half * HALF);
        const uint32_t t_run = tmem + lane_off + RUN_COL + static_cast<uint32_t>(half * HALF);
        const bool last = (c + 1 == nchunks);
        if (EPI == GEMM_DW) {
          // the second of two stacked weights: its constants, its own element count
          const bool second = p.split > 0 && (t / p.num_n) * BM >= p.split;
          n_changed += epi_dw_tile<true, false>(p, second ? p.uc1 : uc,
                                                second ? static_cast<size_t>(p.split) * p.N : 0,
                                                p.dW_out, gm - lane, nbase, HALF / 32, t_acc, xp,
                                                lane);
        } else
#pragma unroll 1
        for (int cc = 0; cc < HALF / 32; ++cc) {
          uint32_t a[32], r[32];
          tmem_ld_32x32b_x32(t_acc + cc * 32, a);
          if (DRAIN && c > 0) tmem_ld_32x32b_x32(t_run + cc * 32, r);
          tmem_ld_wait();
          if (DRAIN && !last) {
            // fold this exact fp32 chunk into the running int32 sum
#pragma unroll
            for (int i = 0; i < 32; ++i)
              r[i] = static_cast<uint32_t>((c > 0 ? static_cast<int32_t>(r[i]) : 0) +
                                           __float2int_rn(__uint_as_float(a[i])));
            tmem_st_32x32b_x32(t_run + cc * 32, r);
            continue;
          }
          const int gn0 = nbase + cc * 32;
          if (gn0 >= p.N) continue;  // warp-uniform
          if (!row_ok) continue;
          if (EPI == GEMM_FWD) epi_fwd(p, gm, gn0, a_t, a, r, DRAIN && c > 0);
          else epi_dx(p, gm, gn0, a);
        }
        if (DRAIN && !last) tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[b]);
      }
    }
    if (!ok && lane == 0) record_timeout(p.status);
    if (EPI == GEMM_DW && p.changed) {
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) n_changed += __shfl_xor_sync(0xffffffffu, n_changed, off);
      if (lane == 0 && n_changed) atomicAdd(p.changed, static_cast<unsigned long long>(n_changed));
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// 2-SM variant (cta_group::2): a cluster of two CTAs on the SM pair of a TPC
// computes a 256 x 256 output tile.  CTA r stages rows [128 r, 128 r + 128)
// of A and rows/columns [128 r, 128 r + 128) of B's 256-wide tile: 32 KB per
// stage instead of 48 KB, so the ring is 7 stages deep (6 for dW, which also
// holds the transpose buffers) and each SM pulls a third fewer operand bytes
// through L2 per FLOP.  Both CTAs' copies complete on the leader's `full`
// barrier; the leader issues the 256 x 256 x 16 MMAs and multicasts its
// commits to both CTAs' `empty` and `acc_full` barriers; each CTA's epilogue
// reads its own 128 rows from its own tensor memory and releases the
// accumulator on the leader's `acc_empty` barrier.
// ---------------------------------------------------------------------------
// Epilogue warps of the 2-SM kernels: the dW update is compute-heavy (AdamW,
// Philox, stochastic rounding per weight) and needs four warps per SM
// sub-partition to hide its latencies; the forward and dX epilogues are light.
template <int EPI, bool DR = false>
struct PairCfg {
  // DR: the exact forward that drains its fp32 accumulator into int32 sums;
  // its folds stall the MMAs, so they are spread over twice the warps
  static constexpr int EW = (EPI == GEMM_DW || DR) ? 16 : 8;
  static constexpr int THREADS = 64 + 32 * EW;
};

template <int EPI, bool DR = false>
struct SmemPair {
  static constexpr int EW = PairCfg<EPI, DR>::EW;
  static constexpr int A_BYTES = 128 * BK * 2;
  static constexpr int B_BYTES = 128 * BK * 2;  // this CTA's half of the B tile
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = (EPI == GEMM_DW) ? 5 : 7;
  static constexpr int XPOSE_OFF = STAGES * STAGE_BYTES;
  static constexpr int XPOSE_BYTES = (EPI == GEMM_DW) ? EW * 32 * kStageLd * 4 : 0;
  static constexpr int BAR_OFF = XPOSE_OFF + XPOSE_BYTES;
  // alignment slack for the 1024-byte swizzle atoms, as much as fits
  static constexpr int SLACK = (232448 - (BAR_OFF + 256)) < 1024 ? (232448 - (BAR_OFF + 256)) : 1024;
  static constexpr int BYTES = BAR_OFF + 256 + SLACK;
  static_assert(SLACK >= 0, "shared memory per CTA");
  static_assert((2 * STAGES + 5) * 8 + 4 <= 176, "barrier area: barriers, then the update constants");
};

// DR (forward only): every chunk of chunk_kb k-blocks is accumulated on its
// own (an exact fp32 integer sum) in the two alternating accumulators, and
// the epilogue warps fold each chunk into running int32 sums held in their
// registers (64 per lane), then write Y from them after the tile's last
// chunk; the MMAs of the next chunk run meanwhile.
// UCD: the dW update constants come from device memory (p.uc_dev, copied to
// shared memory once); otherwise the epilogue reads them straight from the
// kernel's parameter space, where they take no registers.
// GRP: one launch for two dW problems over the same reduction length: p's
// units, then p2's (tensor maps tmA2, tmB2), each with its own shape,
// optimiser state, images, constants and tile order; whole tiles only.
template <bool A_MN, bool B_MN, int EPI, bool PK, bool DR, bool UCD, bool GRP>
__device__ __forceinline__ void gemm_pair_body(const CUtensorMap& tmA, const CUtensorMap& tmB,
                                               const Params& p, const CUtensorMap& tmA2,
                                               const CUtensorMap& tmB2, const Params& p2) {
  using S = SmemPair<EPI, DR>;
  static_assert(!DR || EPI == GEMM_FWD, "drained chunks: exact integer forward only");
  static_assert(!GRP || (EPI == GEMM_DW && !DR && !UCD), "grouped launches: dW, constants by value");
  constexpr int ST = S::STAGES;
  constexpr int EW = S::EW;
  constexpr int BN = 256;           // pair tile width; each CTA holds all 256 columns of its rows
  constexpr int HALF = BN / (EW / 4);  // columns per epilogue warp
  constexpr bool F8 = EPI == GEMM_FWD8;
  constexpr int KB = F8 ? 128 : BK;  // reduction elements per stage (one 128-byte row)
  static_assert(!F8 || (!A_MN && !B_MN), "E4M3 operands are read K-major");
  constexpr uint32_t IDESC = F8 ? idesc_e4m3(256, 256) : idesc_bf16(256, 256, A_MN, B_MN);
  constexpr uint32_t TMEM_COLS = 512;
  constexpr uint32_t MN_CHUNK_BYTES = 64 * BK * 2;

  extern __shared__ uint8_t smem_raw[];
  // The dynamic shared window is 1024-byte aligned in practice; if it is not
  // and the slack cannot absorb it, every CTA of the grid returns here alike.
  if (((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u) > static_cast<uint32_t>(S::SLACK)) {
    if (threadIdx.x == 0) record_timeout(p.status);
    return;
  }
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sA = smem;
  uint8_t* sB = smem + ST * S::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::BAR_OFF);  // used on the leader
  uint64_t* empty = full + ST;
  uint64_t* acc_full = empty + ST;     // [2]
  uint64_t* acc_empty = acc_full + 2;  // [2], used on the leader
  uint64_t* drain_bar = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  // update constants, read by the dW epilogue from shared memory
  UpdateConsts* uc_s = reinterpret_cast<UpdateConsts*>(smem + S::BAR_OFF + 176);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int cid = static_cast<int>(cluster_id_x());
  const int ncl = static_cast<int>(num_clusters_x());

  if (threadIdx.x == 0) {
    for (int s = 0; s < ST; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 2 * EW);
    }
    mbar_init(drain_bar, 1);
    if (EPI == GEMM_DW && UCD) *uc_s = *p.uc_dev;
    fence_mbarrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if (GRP) {
      tma_prefetch_desc(&tmA2);
      tma_prefetch_desc(&tmB2);
    }
  }
  if (warp == 1) tmem_alloc_pair(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers initialised, both allocations done
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t full_lead = mapa_shared(smem_u32(full), 0);
  const uint32_t acc_empty_lead = mapa_shared(smem_u32(acc_empty), 0);

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (both CTAs) ----------------
      int it = 0, s = 0;  // k-blocks issued; stage it % ST
      uint32_t ph = 0;    // phase (it / ST) & 1
      bool ok = true;
      const uint64_t pol_b = EPI == GEMM_DW ? l2_policy_evict_last() : 0ull;
      const uint64_t pol_f = EPI == GEMM_DW ? l2_policy_evict_first() : 0ull;
      // one unit of problem q (tensor maps A, B), its unit index tl; false:
      // a wait ran out
      auto produce = [&](const CUtensorMap& A, const CUtensorMap& B, const Params& q,
                         int tl) -> bool {
        const Unit un = decode_unit(q, tl);
        const int tile = un.tile, kb0 = un.kb0, kb1 = un.kb1;
        const int m0 = pair_tile_m(q, tile) * 256 + static_cast<int>(rank) * 128;
        const int n0 = pair_tile_n(q, tile) * BN + static_cast<int>(rank) * 128;
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          if (it >= ST && !mbar_wait_cl(&empty[s], ph ^ 1u, q.wait_ns)) return false;
          if (leader) mbar_arrive_expect_tx(&full[s], 2 * S::STAGE_BYTES);
          const uint32_t bar = full_lead + 8u * s;
          uint8_t* a = sA + s * S::A_BYTES;
          uint8_t* b = sB + s * S::B_BYTES;
          const int k0 = kb * KB;
          if (!A_MN) {
            tma_load_2d_pair(&A, bar, a, F8 && q.a_wrap ? k0 % q.a_wrap : k0, m0);
          } else if (EPI == GEMM_DW && q.col_major) {
            // column-major tiles: dY's panels are re-read by every wave
#pragma unroll
            for (int j = 0; j < 2; ++j)
              tma_load_2d_pair_hint(&A, bar, a + j * MN_CHUNK_BYTES, m0 + 64 * j, k0, pol_b);
          } else if (EPI == GEMM_DW) {
            // row-major tiles: each dY panel is read by the one wave of
            // clusters that shares it, then never again
#pragma unroll
            for (int j = 0; j < 2; ++j)
              tma_load_2d_pair_hint(&A, bar, a + j * MN_CHUNK_BYTES, m0 + 64 * j, k0, pol_f);
          } else {
#pragma unroll
            for (int j = 0; j < 2; ++j)
              tma_load_2d_pair(&A, bar, a + j * MN_CHUNK_BYTES, m0 + 64 * j, k0);
          }
          if (!B_MN) {
            tma_load_2d_pair(&B, bar, b, k0, n0);
          } else if (EPI == GEMM_DW && !q.col_major) {
            // X~ (all K columns) is re-read by every wave of output-row tiles,
            // while each dY column block is read by one wave: keep X~ in L2
#pragma unroll
            for (int j = 0; j < 2; ++j)
              tma_load_2d_pair_hint(&B, bar, b + j * MN_CHUNK_BYTES, n0 + 64 * j, k0, pol_b);
          } else {
#pragma unroll
            for (int j = 0; j < 2; ++j)
              tma_load_2d_pair(&B, bar, b + j * MN_CHUNK_BYTES, n0 + 64 * j, k0);
          }
          if (++s == ST) {
            s = 0;
            ph ^= 1u;
          }
        }
        return true;
      };
      const int total = GRP ? p.num_tiles + p2.num_tiles : p.num_tiles;
      for (int t = cid; t < total && ok; t += ncl)
        ok = (GRP && t >= p.num_tiles) ? produce(tmA2, tmB2, p2, t - p.num_tiles)
                                       : produce(tmA, tmB, p, t);
      if (!ok) record_timeout(p.status);
      // The leader sees every stage's completion (both CTAs' copies land on
      // its barriers): let the last stages land before the pair exits.
      if (leader)
        for (int i = (it > ST ? it - ST : 0); i < it; ++i)
          mbar_wait_cl(&full[i % ST], (i / ST) & 1u, kDrainNs);
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ---------------- MMA issuer (leader CTA) ----------------
      // The issuing thread shares its scheduler with up to four epilogue
      // warps, so its per-k-block work is kept small: stage index and phase
      // advance incrementally, and the shared-memory descriptors are the
      // stage-0 descriptors plus fixed offsets in their start-address field
      // (address >> 4; every stage lies below 256 KB, so the field never
      // carries into the next one).
      int s = 0;
      uint32_t ph = 0;
      int u = 0;
      bool ok = true;
      const uint64_t a_desc0 = A_MN ? sdesc_sw128(smem_u32(sA), MN_CHUNK_BYTES, 1024)
                                    : sdesc_sw128(smem_u32(sA), 16, 1024);
      const uint64_t b_desc0 = B_MN ? sdesc_sw128(smem_u32(sB), MN_CHUNK_BYTES, 1024)
                                    : sdesc_sw128(smem_u32(sB), 16, 1024);
      // the offsets only change the low word (no carry out of the 14-bit field)
      const uint32_t a_lo0 = static_cast<uint32_t>(a_desc0), b_lo0 = static_cast<uint32_t>(b_desc0);
      const uint64_t a_hi = a_desc0 & 0xFFFFFFFF00000000ull, b_hi = b_desc0 & 0xFFFFFFFF00000000ull;
      constexpr uint32_t kAStage = S::A_BYTES >> 4, kBStage = S::B_BYTES >> 4;
      constexpr uint32_t kAStep = A_MN ? (2048 >> 4) : (32 >> 4);  // per 16-element k step
      constexpr uint32_t kBStep = B_MN ? (2048 >> 4) : (32 >> 4);
      const int total = GRP ? p.num_tiles + p2.num_tiles : p.num_tiles;
      for (int t = cid; t < total && ok; t += ncl) {
        const Unit un =
            (GRP && t >= p.num_tiles) ? decode_unit(p2, t - p.num_tiles) : decode_unit(p, t);
        const int kb0 = un.kb0, kb1 = un.kb1;
        int left = 0;  // DR: k-blocks left in the current chunk
        for (int kb = kb0; kb < kb1; ++kb) {
          // two accumulators alternating per unit; DR: a unit is one chunk of
          // chunk_kb k-blocks, whose exact sum the epilogue folds into int32
          const bool cstart = DR ? left == 0 : kb == kb0;
          if (DR && cstart) left = min(p.chunk_kb, kb1 - kb);
          const int b = u & 1;
          if (cstart && u >= 2) {
            if (!mbar_wait_cl(&acc_empty[b], ((u >> 1) - 1) & 1u, p.wait_ns)) {
              ok = false;
              break;
            }
            tc_fence_after();
          }
          if (!mbar_wait_cl(&full[s], ph, p.wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t alo = a_lo0 + static_cast<uint32_t>(s) * kAStage;
          const uint32_t blo = b_lo0 + static_cast<uint32_t>(s) * kBStage;
          const uint32_t d = tmem + static_cast<uint32_t>(b * BN);
#pragma unroll
          for (int ks = 0; ks < BK / 16; ++ks) {
            const uint32_t acc = (!cstart || ks > 0) ? 1u : 0u;
            const uint64_t ad = a_hi | (alo + ks * kAStep);
            const uint64_t bd = b_hi | (blo + ks * kBStep);
            if (F8) umma_f8_pair(d, ad, bd, IDESC, acc);
            else umma_bf16_pair(d, ad, bd, IDESC, acc);
          }
          umma_commit_pair_mc(&empty[s], 0x3);
          if (++s == ST) {
            s = 0;
            ph ^= 1u;
          }
          if (DR) --left;
          if (kb == kb1 - 1 || (DR && left == 0)) {
            umma_commit_pair_mc(&acc_full[b], 0x3);
            ++u;
          }
        }
      }
      if (!ok) record_timeout(p.status);
      umma_commit_pair(drain_bar);
      mbar_wait_cl(drain_bar, 0, kDrainNs);
    }
  } else {
    // ---------------- epilogue (warps 2 .. EW+1, both CTAs) ----------------
    const int quad = warp & 3;        // tensor-memory lanes this warp may access
    const int half = (warp - 2) >> 2;  // which run of HALF columns
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    float* xp = reinterpret_cast<float*>(smem + S::XPOSE_OFF) + (warp - 2) * 32 * kStageLd;
    uint32_t n_changed = 0, n_changed2 = 0;  // changed codes of p's and p2's units
    int u = 0;
    bool ok = true;
    DwRow st[4];            // dW: optimiser state of the half-chunk being updated
    bool st_loaded = false;  // st already holds this unit's first half-chunk
    // one unit (tile or slice) of problem q, its unit index tl; false: a wait
    // ran out
    auto epi_unit = [&](const Params& q, int tl, uint32_t& n_changed) -> bool {
      const UpdateConsts& uc = UCD ? *uc_s : q.uc;
      const Unit un = decode_unit(q, tl);
      const int tile = un.tile;
      float* dw_out = q.dW_out ? q.dW_out + un.slab * q.slab : nullptr;
      const int gm = pair_tile_m(q, tile) * 256 + static_cast<int>(rank) * 128 + row;
      const int nbase = pair_tile_n(q, tile) * BN + half * HALF;
      const bool row_ok = gm < q.M;
      if (EPI == GEMM_DW && un.slice < 0 && !st_loaded)
        dw_load_first<PK>(q, gm - lane, nbase, lane, st);  // in flight during the wait below
      float a_t = 0.0f;
      if ((EPI == GEMM_FWD || F8) && row_ok) {
        // the second of two stacked weights (whole tiles of columns): its scale
        const float sw = q.split > 0 && pair_tile_n(q, tile) * BN >= q.split ? q.scale1 : q.scale;
        a_t = __fdiv_rn(1.0f, __fmul_rn(q.s_x[gm], sw));
      }
      if (DR) {
        static_assert(!DR || HALF == 64, "two 32-column chunks of running sums per lane");
        const int nchunks = (q.num_kb + q.chunk_kb - 1) / q.chunk_kb;
        int32_t run0[32], run1[32];
        for (int c = 0; c < nchunks; ++c, ++u) {
          const int b = u & 1;
          ok = __all_sync(0xffffffffu, mbar_wait_cl(&acc_full[b], (u >> 1) & 1u, q.wait_ns));
          if (!ok) break;
          tc_fence_after();
          const uint32_t t_acc = tmem + lane_off + static_cast<uint32_t>(b * BN + half * HALF);
          // 16 columns at a time: 64 running sums + 16 loaded values per lane
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint32_t a[16];
            tmem_ld_32x32b_x16(t_acc + 16 * q, a);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              int32_t& rr = q < 2 ? run0[16 * q + i] : run1[16 * (q - 2) + i];
              rr = (c > 0 ? rr : 0) + __float2int_rn(__uint_as_float(a[i]));
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(acc_empty_lead + 8u * b);
        }
        if (!ok) return false;
        if (row_ok) {
          if (nbase < q.N) epi_fwd_int(q, gm, nbase, a_t, run0);
          if (nbase + 32 < q.N) epi_fwd_int(q, gm, nbase + 32, a_t, run1);
        }
        --u;  // the loop header counts one unit per tile
        return true;
      }
      const int b = u & 1;
      ok = __all_sync(0xffffffffu, mbar_wait_cl(&acc_full[b], (u >> 1) & 1u, q.wait_ns));
      if (!ok) return false;
      tc_fence_after();
      const uint32_t t_acc = tmem + lane_off + static_cast<uint32_t>(b * BN + half * HALF);
      if ((EPI == GEMM_DW || EPI == GEMM_FWD || EPI == GEMM_DX) && un.slice >= 0) {
        // a tail slice: its fp32 partial to the slice buffer, tile-local
        // row-major (this lane's row, 32 columns per chunk: 128 contiguous bytes)
        // dW: tile-local row-major (this lane's row, 32 columns per chunk:
        // 128 contiguous bytes), the layout the streaming update reads.
        // Forward / dX: 32 x 32 blocks (block (row / 32, column / 32) at
        // 1024 (8 (row / 32) + column / 32) floats), each stored as [column
        // quad][row][4]: a warp's store of one column quad of its 32 rows is
        // 512 contiguous bytes, and so is the fix-up's load below.
        const int jt = tile - q.full_tiles;
        const long long roff = (static_cast<long long>(rank) * 128 + row) * 256 + half * HALF;
        const long long tile_off = (static_cast<long long>(un.slice) * q.tail_tiles + jt) * 65536LL;
        const int blk0 = ((static_cast<int>(rank) * 4 + quad) * 8 + half * (HALF / 32)) * 1024;
#pragma unroll 1
        for (int cc = 0; cc < HALF / 32; ++cc) {
          uint32_t a[32];
          tmem_ld_32x32b_x32(t_acc + cc * 32, a);
          tmem_ld_wait();
          float4* dst = EPI == GEMM_DW
                            ? reinterpret_cast<float4*>(q.part + tile_off + roff + cc * 32)
                            : reinterpret_cast<float4*>(q.part + tile_off + blk0 + cc * 1024) + lane;
#pragma unroll
          for (int j = 0; j < 8; ++j)
            __stcg(dst + (EPI == GEMM_DW ? j : 32 * j),
                   make_float4(__uint_as_float(a[4 * j]), __uint_as_float(a[4 * j + 1]),
                               __uint_as_float(a[4 * j + 2]), __uint_as_float(a[4 * j + 3])));
        }
        if (EPI == GEMM_FWD || EPI == GEMM_DX) {
          // the last of the tile's slices to finish this warp's region adds
          // the partials in slice order and applies the epilogue
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(acc_empty_lead + 8u * b);  // accumulator released
          __threadfence();
          __syncwarp();
          unsigned long long done = 0;
          if (lane == 0) {
            unsigned long long* ctr =
                q.tail_ctr + (static_cast<long long>(jt) * 2 + rank) * EW + (warp - 2);
            unsigned long long assumed = 0ull, nv;
            while (true) {  // at most tail_splits + 1 tries: each failure sees another slice's count
              nv = (assumed >> 16) == q.tail_tag ? assumed + 1ull : ((q.tail_tag << 16) | 1ull);
              const unsigned long long prev = atomicCAS(ctr, assumed, nv);
              if (prev == assumed) break;
              assumed = prev;
            }
            done = nv & 0xFFFFull;
          }
          done = __shfl_sync(0xffffffffu, done, 0);
          if (done == static_cast<unsigned long long>(q.tail_splits)) {
            __threadfence();
            const float* src0 = q.part + static_cast<long long>(jt) * 65536LL + blk0;
            const long long sstride = static_cast<long long>(q.tail_tiles) * 65536LL;
#pragma unroll 1
            for (int cc = 0; cc < HALF / 32; ++cc) {
              const int gn0 = nbase + cc * 32;
              float f[32];
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                const float4 v = __ldcg(reinterpret_cast<const float4*>(src0 + cc * 1024) + 32 * j + lane);
                f[4 * j] = v.x;
                f[4 * j + 1] = v.y;
                f[4 * j + 2] = v.z;
                f[4 * j + 3] = v.w;
              }
#pragma unroll 1
              for (int sl = 1; sl < q.tail_splits; ++sl) {
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                  const float4 v = __ldcg(
                      reinterpret_cast<const float4*>(src0 + sl * sstride + cc * 1024) + 32 * j + lane);
                  f[4 * j] = __fadd_rn(f[4 * j], v.x);
                  f[4 * j + 1] = __fadd_rn(f[4 * j + 1], v.y);
                  f[4 * j + 2] = __fadd_rn(f[4 * j + 2], v.z);
                  f[4 * j + 3] = __fadd_rn(f[4 * j + 3], v.w);
                }
              }
              // every slice's block of this chunk is read: drop its lines
              // from L2 so that they are never written back
              __syncwarp();
#pragma unroll 1
              for (int sl = 0; sl < q.tail_splits; ++sl)
                l2_discard_line(src0 + sl * sstride + cc * 1024 + lane * 32);
              if (gn0 >= q.N || !row_ok) continue;
              uint32_t a[32];
#pragma unroll
              for (int i = 0; i < 32; ++i) a[i] = __float_as_uint(f[i]);
              if (EPI == GEMM_FWD) epi_fwd(q, gm, gn0, a_t, a, a, false);  // no running sums
              else epi_dx(q, gm, gn0, a);
            }
          }
          return true;  // the accumulator is already released
        }
      } else if (EPI == GEMM_DW) {
        // the first half-chunk of this warp's next unit, if a whole tile,
        // is loaded during this tile's last half-chunk
        int row0n = -1, nbasen = 0;
        if (tl + ncl < q.num_tiles) {
          const Unit nu = decode_unit(q, tl + ncl);
          if (nu.slice < 0) {
            row0n = pair_tile_m(q, nu.tile) * 256 + static_cast<int>(rank) * 128 + quad * 32;
            nbasen = pair_tile_n(q, nu.tile) * BN + half * HALF;
          }
        }
        // the second of two stacked weights: its constants, its own element count
        if (q.split > 0 && pair_tile_m(q, tile) * 256 >= q.split)
          n_changed += epi_dw_tile_roll<PK, !UCD>(q, q.uc1, q.pc1, static_cast<size_t>(q.split) * q.N,
                                                  dw_out, gm - lane, nbase, HALF / 32, t_acc, xp,
                                                  lane, st, row0n, nbasen);
        else
          n_changed += epi_dw_tile_roll<PK, !UCD>(q, uc, q.pc, 0, dw_out, gm - lane, nbase,
                                                  HALF / 32, t_acc, xp, lane, st, row0n, nbasen);
        st_loaded = row0n >= 0;
      } else
#pragma unroll 1
      for (int cc = 0; cc < HALF / 32; ++cc) {
        uint32_t a[32], r[32];
        tmem_ld_32x32b_x32(t_acc + cc * 32, a);
        tmem_ld_wait();
        const int gn0 = nbase + cc * 32;
        if (gn0 >= q.N) continue;  // warp-uniform
        if (!row_ok) continue;
        if (EPI == GEMM_FWD) epi_fwd(q, gm, gn0, a_t, a, r, false);
        else if (F8) epi_fwd8(q, gm, gn0, a_t, a);
        else epi_dx(q, gm, gn0, a);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(acc_empty_lead + 8u * b);
      return true;
    };
    const int total = GRP ? p.num_tiles + p2.num_tiles : p.num_tiles;
    for (int t = cid; t < total && ok; t += ncl, ++u)
      ok = (GRP && t >= p.num_tiles) ? epi_unit(p2, t - p.num_tiles, n_changed2)
                                     : epi_unit(p, t, n_changed);
    if (!ok && lane == 0) record_timeout(p.status);
    if (EPI == GEMM_DW && p.changed) {
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) n_changed += __shfl_xor_sync(0xffffffffu, n_changed, off);
      if (lane == 0 && n_changed) atomicAdd(p.changed, static_cast<unsigned long long>(n_changed));
    }
    if (GRP && p2.changed) {
#pragma unroll
      for (int off = 16; off > 0; off >>= 1)
        n_changed2 += __shfl_xor_sync(0xffffffffu, n_changed2, off);
      if (lane == 0 && n_changed2) atomicAdd(p2.changed, static_cast<unsigned long long>(n_changed2));
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no remote arrive, copy or MMA of either CTA is pending
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, TMEM_COLS);
  }
}

template <bool A_MN, bool B_MN, int EPI, bool PK = false, bool DR = false, bool UCD = false>
__global__ void __launch_bounds__(PairCfg<EPI, DR>::THREADS, 1)
    gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA,
                     const __grid_constant__ CUtensorMap tmB, const __grid_constant__ Params p) {
  gemm_pair_body<A_MN, B_MN, EPI, PK, DR, UCD, false>(tmA, tmB, p, tmA, tmB, p);
}

// Two dW + update problems in one persistent launch (both operands MN-major,
// int8 codes, constants by value).
__global__ void __launch_bounds__(PairCfg<GEMM_DW, false>::THREADS, 1)
    gemm_dw_group_kernel(const __grid_constant__ CUtensorMap tmA,
                         const __grid_constant__ CUtensorMap tmB, const __grid_constant__ Params p,
                         const __grid_constant__ CUtensorMap tmA2,
                         const __grid_constant__ CUtensorMap tmB2,
                         const __grid_constant__ Params p2) {
  gemm_pair_body<true, true, GEMM_DW, false, false, false, true>(tmA, tmB, p, tmA2, tmB2, p2);
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

// 2-D row-major matrix of 2-byte (bf16) or 1-byte (E4M3) elements with
// `inner` contiguous elements per row and `outer` rows; box of box_inner x
// box_outer, 128-byte swizzle, zero fill.
bool make_map(CUtensorMap* map, const void* ptr, uint64_t inner, uint64_t outer,
              uint32_t box_inner, uint32_t box_outer, int elem_bytes = 2, uint64_t row_elems = 0) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  // The encoder is a driver call and needs a context current in the calling
  // thread.  A thread whose first CUDA work in this process comes through
  // this library (an autograd worker running a backward, say) may not have
  // one bound yet: a runtime call binds the device's primary context.
  thread_local bool bound = false;
  if (!bound) {
    if (cudaFree(nullptr) != cudaSuccess) return false;
    bound = true;
  }
  const cuuint64_t dims[2] = {inner, outer};
  // rows `row_elems` elements apart (0: packed rows of `inner`)
  const cuuint64_t strides[1] = {(row_elems ? row_elems : inner) * static_cast<cuuint64_t>(elem_bytes)};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, elem_bytes == 1 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
             2, const_cast<void*>(ptr), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, bool A_MN, bool B_MN, int EPI, bool DRAIN>
int launch_tiles(const CUtensorMap& ta, const CUtensorMap& tb, Params p, cudaStream_t stream) {
  auto kern = gemm_kernel<BN, A_MN, B_MN, EPI, DRAIN>;
  const int smem = Smem<BN, EPI>::BYTES;
  static bool attr_set = false;  // per template instance
  if (!attr_set) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
        cudaSuccess)
      return 3;
    attr_set = true;
  }
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  p.num_n = (p.N + BN - 1) / BN;
  p.num_tiles = ((p.M + BM - 1) / BM) * p.num_n;
  const int grid = p.num_tiles < sms ? p.num_tiles : sms;
  kern<<<grid, kThreads, smem, stream>>>(ta, tb, p);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

template <bool A_MN, bool B_MN, int EPI, bool PK = false, bool DR = false, bool UCD = false>
int launch_pairs(const CUtensorMap& ta, const CUtensorMap& tb, Params p, cudaStream_t stream,
                 void* tail_ws = nullptr, size_t tail_ws_bytes = 0, TailPlan* plan = nullptr);

}  // namespace

// Tail of a 2-SM dW GEMM on `clusters` clusters: the tiles past the last
// full wave are cut into S token slices (about `clusters` units in the last
// wave, each slice at least 4 k-blocks long, S <= 16), so that the last wave
// costs a fraction of a tile's reduction, and their update moves out of the
// GEMM's epilogue into a streaming kernel.
TailPlan tail_plan(int M, int N, int Kred, int clusters) {
  TailPlan t{0, 0, 0, 0, 0};
  const int tiles = ((M + 255) / 256) * ((N + 255) / 256);
  const int num_kb = (Kred + BK - 1) / BK;
  if (clusters < 2) return t;
  const int full = (tiles / clusters) * clusters;
  const int tail = tiles - full;
  if (full == 0 || tail == 0) return t;
  int S = clusters / tail;
  if (S > num_kb / 4) S = num_kb / 4;
  if (S > 16) S = 16;
  if (S < 2) return t;
  const int kbps = (num_kb + S - 1) / S;
  S = (num_kb + kbps - 1) / kbps;  // no empty slice
  if (S < 2) return t;
  t.splits = S;
  t.tail = tail;
  t.full = full;
  t.kbps = kbps;
  t.bytes = static_cast<size_t>(tail) * S * 65536 * sizeof(float);
  return t;
}

// Forward / dX tail workspace: the slice counters (2 CTA ranks x 8 epilogue
// warps per tail tile, tail <= clusters) in the first kTailCtrBytes, then the
// partials (tail * splits <= clusters tiles of 256 x 256 floats).
constexpr size_t kTailCtrBytes = 16384;

// The tail partials start on a 256-byte boundary inside the workspace (the
// consumers discard each 128-byte line from L2 once read, which must not
// touch a neighbour's bytes); the size functions leave 256 bytes for it.
static float* tail_partials(void* ws, size_t ctr) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(ws) + ctr;
  return reinterpret_cast<float*>((a + 255) & ~static_cast<uintptr_t>(255));
}

// A forward or dX GEMM cuts its last wave only when the reduction is at
// least 4096 long: a slice's fixed costs (its pipeline fill, the partials'
// round trip through L2, the fix-up) are ~10 us, which a cut of a 2048-long
// reduction (~12 us of tile) does not win back.
constexpr int kTailMinKb = 4096 / BK;

size_t gemm_tail_bytes(int M, int N, int Kred) {
  if ((Kred + BK - 1) / BK < kTailMinKb) return 0;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const TailPlan tp = tail_plan(M, N, Kred, sms / 2);
  // any launch's plan has tail * splits <= its clusters <= sms / 2
  return tp.splits >= 2 ? kTailCtrBytes + 256 + static_cast<size_t>(sms / 2) * 65536 * sizeof(float)
                        : 0;
}

// Token slices for a 2-SM dW GEMM whose output tiles would leave most SM
// pairs idle: enough slices to give every pair a unit of work, each slice at
// least 4 k-blocks (256 tokens) long, at most 32 slices.
int dw_splits(int M, int N, int Kred) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int pairs = sms / 2;
  const long long tiles = static_cast<long long>((M + 255) / 256) * ((N + 255) / 256);
  const int num_kb = (Kred + BK - 1) / BK;
  if (tiles * 2 > pairs || num_kb < 8) return 1;
  long long s = pairs / tiles;
  if (s > num_kb / 4) s = num_kb / 4;
  if (s > 32) s = 32;
  return s < 2 ? 1 : static_cast<int>(s);
}

namespace {

// Launches that cut their last wave with slice counters (all GEMM kinds).
std::atomic<unsigned long long> g_tail_launches{0};

// 256 x 256 pair tiles of a 2-SM launch.  dW: the operand with fewer
// 256-wide panels is the one re-read by every wave (and kept in L2): X_tilde
// (along the rows) when the output has more row tiles, dY (down the columns)
// when it has more column tiles.
void pair_tiling(Params& p, bool dw) {
  p.num_n = (p.N + 255) / 256;
  p.num_m = (p.M + 255) / 256;
  p.num_tiles = p.num_m * p.num_n * p.splits;
  p.col_major = dw && p.num_n > p.num_m;
}

template <bool A_MN, bool B_MN, int EPI, bool PK, bool DR, bool UCD>
int launch_pairs(const CUtensorMap& ta, const CUtensorMap& tb, Params p, cudaStream_t stream,
                 void* tail_ws, size_t tail_ws_bytes, TailPlan* plan) {
  auto kern = gemm_pair_kernel<A_MN, B_MN, EPI, PK, DR, UCD>;
  const int smem = SmemPair<EPI, DR>::BYTES;
  constexpr int threads = PairCfg<EPI, DR>::THREADS;
  static int max_clusters = 0;  // per template instance
  pair_tiling(p, EPI == GEMM_DW);
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(threads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (max_clusters == 0) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
        cudaSuccess)
      return 3;
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    cfg.gridDim = dim3(sms, 1, 1);
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n < 1) return 3;
    max_clusters = n;
  }
  p.full_units = p.num_tiles;
  p.full_tiles = p.num_tiles;
  p.tail_tiles = 0;
  p.tail_splits = 1;
  p.tail_kbps = p.num_kb;
  p.part = nullptr;
  if (plan) *plan = TailPlan{0, 0, 0, 0, 0};
  if ((EPI == GEMM_DW || ((EPI == GEMM_FWD || EPI == GEMM_DX) && !DR && p.num_kb >= kTailMinKb)) &&
      tail_ws && plan && p.splits == 1) {
    const TailPlan tp = tail_plan(p.M, p.N, p.Kred, max_clusters);
    const size_t ctr = EPI == GEMM_DW ? 0 : kTailCtrBytes;
    static_assert(2 * 8 * 8 * 128 <= kTailCtrBytes, "slice counters: 128 tail tiles");
    float* part = tail_partials(tail_ws, ctr);
    const size_t used = static_cast<size_t>(reinterpret_cast<uint8_t*>(part) -
                                            static_cast<uint8_t*>(tail_ws)) + tp.bytes;
    if (tp.splits >= 2 && tp.tail <= 128 && used <= tail_ws_bytes) {
      p.full_units = tp.full;
      p.full_tiles = tp.full;
      p.tail_tiles = tp.tail;
      p.tail_splits = tp.splits;
      p.tail_kbps = tp.kbps;
      p.part = part;
      p.num_tiles = tp.full + tp.tail * tp.splits;
      if (EPI != GEMM_DW) {
        // The launch's tag: the process's count of such launches (one count
        // for every GEMM kind, so a forward's counters never carry a later
        // dX launch's tag), spread over 47 bits by an odd multiplier
        // (distinct for distinct counts below 2^47), with bit 47 set, so
        // that no word a workspace held before -- a small integer such as a
        // count, or a positive float -- reads as this launch's tag.
        const unsigned long long n = g_tail_launches.fetch_add(1) + 1;
        p.tail_ctr = static_cast<unsigned long long*>(tail_ws);
        p.tail_tag = ((n * 0x9E3779B97F4A7C15ull) & 0x7FFFFFFFFFFFull) | 0x800000000000ull;
      }
      *plan = tp;
    }
  }
  const int clusters = p.num_tiles < max_clusters ? p.num_tiles : max_clusters;
  cfg.gridDim = dim3(2 * clusters, 1, 1);
  if (cudaLaunchKernelEx(&cfg, kern, ta, tb, p) != cudaSuccess) return 3;
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

}  // namespace

// The per-call Philox constants of PhiloxCall from the update constants.
static PhiloxCall philox_call_consts(const UpdateConsts& uc) {
  PhiloxCall k{};
  for (int r = 0; r < 10; ++r) {
    k.rk[2 * r] = uc.key0 + static_cast<uint32_t>(r) * 0x9E3779B9u;
    k.rk[2 * r + 1] = uc.key1 + static_cast<uint32_t>(r) * 0xBB67AE85u;
  }
  const uint64_t p1 = static_cast<uint64_t>(0xCD9E8D57u) * uc.step_lo;
  k.c0x = static_cast<uint32_t>(p1 >> 32) ^ k.rk[0];
  k.c0y = static_cast<uint32_t>(p1);
  k.x3k = uc.tensor_id ^ k.rk[1];
  return k;
}

// The arguments every GEMM kind takes from its launch record (the watchdog,
// pointers, scales, update constants and images).
static int fill_common(const GemmLaunch& g, Params& p) {
  p.wait_ns = wait_limit_ns();
  p.status = status_word();
  if (!p.status) return 3;
  p.s_x = g.s_x;
  p.scale = g.scale;
  p.out_bf16 = static_cast<__nv_bfloat16*>(g.out_bf16);
  p.acc_out = g.acc_out;
  p.acc_f32 = g.acc_f32;
  p.W = g.W;
  p.packed = g.packed;
  p.m = g.m;
  p.v = g.v;
  p.dW_out = g.dW_out;
  p.changed = g.changed;
  p.uc = g.uc;
  p.pc = philox_call_consts(g.uc);
  p.uc_dev = g.uc_dev;
  p.split = g.split;
  p.scale1 = g.scale1;
  p.uc1 = g.uc1;
  p.pc1 = philox_call_consts(g.uc1);
  p.img_next = g.kind == GEMM_DW ? static_cast<__nv_bfloat16*>(g.img_next) : nullptr;
  p.img8_next = g.kind == GEMM_DW ? static_cast<uint8_t*>(g.img8_next) : nullptr;
  p.img8_split = p.img8_next && g.img8_split ? 1 : 0;
  p.a_wrap = g.kind == GEMM_FWD8 ? g.a_wrap : 0;
  if ((p.img_next || p.img8_next) && (g.packed || !g.W)) return 1;
  return 0;
}

int launch_gemm(const GemmLaunch& g, cudaStream_t stream) {
  Params p{};
  p.M = g.M;
  p.N = g.N;
  p.Kred = g.Kred;
  const int kb_elems = g.kind == GEMM_FWD8 ? 128 : BK;
  p.num_kb = (g.Kred + kb_elems - 1) / kb_elems;
  p.chunk_kb = p.num_kb;
  if (g.kind == GEMM_FWD) {
    const int ck = g.chunk_k / BK;
    if (ck < 1) return 1;
    if (ck < p.num_kb) p.chunk_kb = ck;
  }
  const bool drain = p.chunk_kb < p.num_kb;
  GemmLaunch gl = g;
  // packed codes: the 2-SM kernel whatever the tiling mode
  gl.pair = !drain && (gemm_mode() == 0 || g.packed);
  const GemmLaunch& g2 = gl;
  p.splits = 1;
  p.kb_per_split = p.num_kb;
  p.slab = 0;
  int splits = 1;
  if (g.kind == GEMM_DW && g2.pair && g.ws)
    splits = dw_splits(g.M, g.N, g.Kred);
  if (splits > 1 && g.ws_bytes >= static_cast<size_t>(splits) * g.M * g.N * sizeof(float)) {
    p.kb_per_split = (p.num_kb + splits - 1) / splits;
    p.splits = (p.num_kb + p.kb_per_split - 1) / p.kb_per_split;
    p.slab = static_cast<long long>(g.M) * g.N;
  }
  const int rc = fill_common(g, p);
  if (rc) return rc;
  // stacked weights: whole tiles (multiples of 256 of either tiling),
  // constants in the parameter space
  if (g.split > 0 && (g.split % 256 != 0 || g.uc_dev ||
                      (g.kind != GEMM_FWD && g.kind != GEMM_FWD8 && g.kind != GEMM_DW) ||
                      g.split >= (g.kind == GEMM_DW ? g.M : g.N)))
    return 1;

  CUtensorMap ta, tb;
  switch (g.kind) {
    case GEMM_FWD:
      if (!make_map(&ta, g.A, g.Kred, g.M, BK, BM)) return 3;
      if (drain) {
        if (!make_map(&tb, g.B, g.Kred, g.N, BK, 128)) return 3;
        if (gemm_mode() == 0)
          return launch_pairs<false, false, GEMM_FWD, false, true>(ta, tb, p, stream);
        return launch_tiles<128, false, false, GEMM_FWD, true>(ta, tb, p, stream);
      }
      if (!make_map(&tb, g.B, g.Kred, g.N, BK, g2.pair ? 128 : 256)) return 3;
      if (g2.pair) {
        // with a workspace, the last wave's tiles as reduction slices
        TailPlan tp{0, 0, 0, 0, 0};
        return launch_pairs<false, false, GEMM_FWD>(ta, tb, p, stream, g.ws, g.ws_bytes,
                                                    g.ws ? &tp : nullptr);
      }
      return launch_tiles<256, false, false, GEMM_FWD, false>(ta, tb, p, stream);
    case GEMM_FWD8:
      // 2-SM tiles whatever the tiling mode: E4M3 rows of 128 elements
      if (g.a_wrap && (g.a_wrap % 128 != 0 || g.Kred != 2 * g.a_wrap)) return 1;
      if (!make_map(&ta, g.A, g.a_wrap ? g.a_wrap : g.Kred, g.M, 128, BM, 1)) return 3;
      if (!make_map(&tb, g.B, g.Kred, g.N, 128, 128, 1)) return 3;
      return launch_pairs<false, false, GEMM_FWD8>(ta, tb, p, stream);
    case GEMM_DX:
      if (!make_map(&ta, g.A, g.Kred, g.M, BK, BM, 2, static_cast<uint64_t>(g.lda))) return 3;
      if (!make_map(&tb, g.B, g.N, g.Kred, 64, BK)) return 3;
      if (g2.pair) {
        TailPlan tp{0, 0, 0, 0, 0};
        return launch_pairs<false, true, GEMM_DX>(ta, tb, p, stream, g.ws, g.ws_bytes,
                                                  g.ws ? &tp : nullptr);
      }
      return launch_tiles<256, false, true, GEMM_DX, false>(ta, tb, p, stream);
    case GEMM_DW: {
      if (!make_map(&ta, g.A, g.M, g.Kred, 64, BK)) return 3;
      if (!make_map(&tb, g.B, g.N, g.Kred, 64, BK)) return 3;
      if (!g2.pair) return launch_tiles<256, true, true, GEMM_DW, false>(ta, tb, p, stream);
      if (p.splits == 1) {
        // the last wave's tiles as token slices, their update in a streaming pass
        TailPlan tp{0, 0, 0, 0, 0};
        const bool pk = p.packed && p.W;
        const bool ucd = p.uc_dev != nullptr;
        const int rc =
            pk ? (ucd ? launch_pairs<true, true, GEMM_DW, true, false, true>(ta, tb, p, stream,
                                                                             g.ws, g.ws_bytes, &tp)
                      : launch_pairs<true, true, GEMM_DW, true>(ta, tb, p, stream, g.ws,
                                                                g.ws_bytes, &tp))
               : (ucd ? launch_pairs<true, true, GEMM_DW, false, false, true>(
                            ta, tb, p, stream, g.ws, g.ws_bytes, &tp)
                      : launch_pairs<true, true, GEMM_DW>(ta, tb, p, stream, g.ws, g.ws_bytes,
                                                          &tp));
        if (rc || tp.splits == 0) return rc;
        return launch_tail_update(tail_partials(g.ws, 0), tp.splits, tp.tail, tp.full,
                                  (g.N + 255) / 256, g.M, g.N, g.W, g.packed, g.m, g.v, g.uc,
                                  g.uc_dev, g.changed, g.dW_out, stream,
                                  g.split > 0 ? &g.uc1 : nullptr, g.split,
                                  (g.N + 255) / 256 > (g.M + 255) / 256,
                                  static_cast<uint16_t*>(g.img_next),
                                  static_cast<uint8_t*>(g.img8_next), p.img8_split != 0);
      }
      // split-T: fp32 partials of each token slice into the workspace slabs,
      // then one streaming pass sums the slabs in slice order and applies the
      // AdamW + stochastic-rounding update (and writes the summed gradient to
      // dW_out if asked for)
      Params ps = p;
      ps.W = nullptr;
      ps.m = nullptr;
      ps.v = nullptr;
      ps.changed = nullptr;
      ps.dW_out = static_cast<float*>(g.ws);
      const int rc = launch_pairs<true, true, GEMM_DW>(ta, tb, ps, stream);
      if (rc) return rc;
      if (!g.W) {
        // gradient only: sum the slabs into dW_out
        return launch_slab_sum(static_cast<const float*>(g.ws), p.splits, p.slab, g.dW_out,
                               stream);
      }
      // (the images of the updated codes are written by the same pass)
      uint16_t* img = static_cast<uint16_t*>(g.img_next);
      uint8_t* img8 = static_cast<uint8_t*>(g.img8_next);
      const int64_t img8_k = p.img8_split ? g.N : 0;  // split image rows: 2 N bytes
      if (g.split > 0) {
        // stacked weights: the rows of each with its own constants
        const long long n0 = static_cast<long long>(g.split) * g.N;
        const float* sl = static_cast<const float*>(g.ws);
        return launch_sr_update_slabs(sl, p.splits, p.slab, g.W, g.m, g.v, n0, g.uc, nullptr,
                                      g.changed, g.dW_out, stream, g.packed, img, img8, img8_k) ||
               launch_sr_update_slabs(sl + n0, p.splits, p.slab, g.W + n0, g.m + n0, g.v + n0,
                                      p.slab - n0, g.uc1, nullptr, g.changed,
                                      g.dW_out ? g.dW_out + n0 : nullptr, stream, g.packed,
                                      img ? img + n0 : nullptr,
                                      img8 ? img8 + (img8_k ? 2 * n0 : n0) : nullptr, img8_k);
      }
      return launch_sr_update_slabs(static_cast<const float*>(g.ws), p.splits, p.slab, g.W, g.m,
                                    g.v, p.slab, g.uc, g.uc_dev, g.changed, g.dW_out, stream,
                                    g.packed, img, img8, img8_k);
    }
  }
  return 1;
}

int launch_dw_group(const GemmLaunch& g0, const GemmLaunch& g1, cudaStream_t stream) {
  if (g0.kind != GEMM_DW || g1.kind != GEMM_DW || g0.Kred != g1.Kred) return 1;
  Params p[2];
  CUtensorMap ta[2], tb[2];
  for (int i = 0; i < 2; ++i) {
    const GemmLaunch& g = i ? g1 : g0;
    if (g.packed || !g.W || !g.m || !g.v || g.uc_dev) return 1;
    if (g.split > 0 && (g.split % 256 != 0 || g.split >= g.M)) return 1;
    Params& q = p[i];
    q = Params{};
    q.M = g.M;
    q.N = g.N;
    q.Kred = g.Kred;
    q.num_kb = (g.Kred + BK - 1) / BK;
    q.chunk_kb = q.num_kb;
    q.splits = 1;
    q.kb_per_split = q.num_kb;
    q.slab = 0;
    const int rc = fill_common(g, q);
    if (rc) return rc;
    pair_tiling(q, true);
    // whole tiles only: the two problems' tiles fill the waves together
    q.full_units = q.num_tiles;
    q.full_tiles = q.num_tiles;
    q.tail_tiles = 0;
    q.tail_splits = 1;
    q.tail_kbps = q.num_kb;
    q.part = nullptr;
    if (!make_map(&ta[i], g.A, g.M, g.Kred, 64, BK)) return 3;
    if (!make_map(&tb[i], g.B, g.N, g.Kred, 64, BK)) return 3;
  }
  auto kern = gemm_dw_group_kernel;
  const int smem = SmemPair<GEMM_DW, false>::BYTES;
  constexpr int threads = PairCfg<GEMM_DW, false>::THREADS;
  static int max_clusters = 0;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(threads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (max_clusters == 0) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
        cudaSuccess)
      return 3;
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    cfg.gridDim = dim3(sms, 1, 1);
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n < 1) return 3;
    max_clusters = n;
  }
  const int total = p[0].num_tiles + p[1].num_tiles;
  const int clusters = total < max_clusters ? total : max_clusters;
  cfg.gridDim = dim3(2 * clusters, 1, 1);
  if (cudaLaunchKernelEx(&cfg, kern, ta[0], tb[0], p[0], ta[1], tb[1], p[1]) != cudaSuccess)
    return 3;
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

}  // namespace dqt

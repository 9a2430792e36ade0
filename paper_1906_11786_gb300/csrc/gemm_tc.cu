// Split-K "TN" GEMM on tcgen05 for the weight-gradient reductions of the backward pass:
//     part[s][m][n] = sum_{k in split s} A[m][k] B[n][k]        (A, B bf16, K contiguous; fp32)
// followed by a deterministic reduction over the splits into the gradient layout.  The weight
// gradients of Eq. 1's transforms and of the GRU are sums over every node (and every step) of
// outer products, i.e. exactly such GEMMs with K = nodes; their bias gradients come out of the
// same product through a row of ones appended to B.
//
// 192 threads: warp 0 issues TMA loads into a 4-stage ring, warp 1 allocates TMEM and issues the
// MMAs (lane 0), warps 2-5 read the accumulator back (one TMEM lane quarter each).
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>

#include "gemm_tc.h"
#include "kernels.h"
#include "tc_util.cuh"

namespace bg {

using namespace tc;

namespace {

constexpr int kStages = 4;

// Tile widths BN = Hout + 16 (48, 80, 144, 272), four stages each, one CTA per SM.  A CTA takes
// MT = 2 consecutive 128-row M tiles of one problem (MT = 1 at BN = 272, whose accumulator takes all
// 512 TMEM columns), so that each K chunk of B, which every M tile of the problem reads, is loaded
// once per two tiles: the pass moves A once and B once per tile pair, instead of once per tile.
// B is [X^T; 1; 0]: its Hout = BN - 16 data rows come by TMA (one box of at most 256 rows), and
// its last 16 rows, a ones row (the bias column of the product) and zeros, are the same for every K
// chunk, so the kernel writes them once into each stage at its start.  BN = 272 issues an N = 256
// and an N = 16 MMA per K step.
template <int BN>
struct GCfg {
  static constexpr int MT = BN <= 256 ? 2 : 1;
  static constexpr int A_BYTES = 128 * 128;  // 128 rows x 64 bf16
  static constexpr int B_BYTES = BN * 128;
  static constexpr int STAGE = MT * A_BYTES + B_BYTES;
  static constexpr int STAGES = 4;
  static constexpr int SMEM = STAGES * STAGE + 1024 + 1024;
  static constexpr int TCOLS = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : BN <= 256 ? 256 : 512;
  static constexpr int BROWS = BN - 16;                 // B rows loaded per K chunk (one box)
  static constexpr int N1 = BN <= 256 ? BN : 256;      // first MMA's N
  static_assert(BN % 16 == 0 && BN <= 512, "tile width");
  static_assert(SMEM + 512 <= 232448, "shared memory");
  static_assert(MT * TCOLS <= 512, "tensor memory");
  static_assert(BROWS <= 256 && BROWS * 128 % 1024 == 0 && A_BYTES % 1024 == 0, "box alignment");
  static_assert(STAGES <= kStages, "stage count");
};

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

// Up to kMaxGroups problems with the same K and N in one launch: blockIdx.x runs over the work
// items (MT consecutive M tiles of one problem) of all groups; group g's rows sit at rows
// prow[g] .. prow[g] + M[g] of the partial sums.
constexpr int kMaxGroups = 4;
struct TNGroups {
  CUtensorMap a[kMaxGroups], b[kMaxGroups];
  int it_end[kMaxGroups];  // cumulative work-item counts
  int M[kMaxGroups];
  int prow[kMaxGroups];
};

template <int BN>
__global__ void __launch_bounds__(192, 1)
    k_gemm_tn(const __grid_constant__ TNGroups grp, float* __restrict__ part, int Mtot, int N,
              int kchunks, int per_split, int* status) {
  using C = GCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE);
  uint64_t* empty = full + C::STAGES;
  uint64_t* done = empty + C::STAGES;
  uint64_t* drain = done + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
  volatile int* abort = abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int g = 0;
  while (g + 1 < kMaxGroups && (int)blockIdx.x >= grp.it_end[g]) ++g;
  const int item = blockIdx.x - (g ? grp.it_end[g - 1] : 0), split = blockIdx.z;
  const int M = grp.M[g];
  const int mt0 = item * C::MT;                            // first M tile of this CTA
  const int ntiles = min(C::MT, (M + 127) / 128 - mt0);    // 1 .. MT
  const CUtensorMap* tmA = &grp.a[g];
  const CUtensorMap* tmB = &grp.b[g];
  const int kc0 = split * per_split;
  const int kc1 = min(kchunks, kc0 + per_split);
  // the last 16 rows of every stage's B: row Hout all bf16 ones, the rest zeros (128 bytes a row;
  // all 16-byte chunks of a row equal, so the 128-byte swizzle leaves them in place)
  for (int i = threadIdx.x; i < C::STAGES * 16 * 8; i += blockDim.x) {
    const int s = i / 128, r = (i / 8) % 16, c = i % 8;
    const uint32_t v = r == 0 ? 0x3F803F80u : 0u;
    *reinterpret_cast<uint4*>(smem + s * C::STAGE + C::MT * C::A_BYTES + (C::BROWS + r) * 128 + c * 16) =
        make_uint4(v, v, v, v);
  }
  fence_proxy_async();  // visible to the tensor cores' shared-memory reads
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(done, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::MT * C::TCOLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  grid_dep_launch();  // TMEM is held: the reduction may be scheduled as SMs free up
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(tmA);
    tma_prefetch_desc(tmB);
    grid_dep_wait();  // A and B are the previous kernels' output
    uint32_t issued[kStages] = {0, 0, 0, 0};
    for (int kc = kc0, it = 0; kc < kc1; ++kc, ++it) {
      const int s = it % C::STAGES;
      if (!mbar_wait(&empty[s], ((it / C::STAGES) & 1) ^ 1, status, 501, abort, 32)) break;
      ++issued[s];
      mbar_expect_tx(&full[s], ntiles * C::A_BYTES + C::BROWS * 128);
      uint8_t* st = smem + s * C::STAGE;
      for (int m = 0; m < ntiles; ++m)
        tma_load_2d(st + m * C::A_BYTES, tmA, &full[s], kc * 64, (mt0 + m) * 128);
      tma_load_2d(st + C::MT * C::A_BYTES, tmB, &full[s], kc * 64, blockIdx.y * BN);
    }
    if (*abort)
      for (int s = 0; s < C::STAGES; ++s)
        for (uint32_t t = 0; issued[s] && t < (1u << 22) && !mbar_try(&full[s], (issued[s] - 1) & 1); ++t) {
        }
  } else if (warp == 1) {
    // the whole warp runs the loop (uniform operands); one elected lane issues
    const bool leader = elect_one_sync();
    constexpr uint32_t idesc = idesc_bf16_f32(128, C::N1);
    constexpr uint32_t idesc2 = idesc_bf16_f32(128, BN > 256 ? BN - 256 : 16);
    for (int kc = kc0, it = 0; kc < kc1; ++kc, ++it) {
      const int s = it % C::STAGES;
      if (!mbar_wait(&full[s], (it / C::STAGES) & 1, status, 502, abort)) break;
      tc_fence_after();
      const uint32_t a = smem_u32(smem + s * C::STAGE), b = a + C::MT * C::A_BYTES;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        if (leader) {
          const uint32_t acc = (kc > kc0 || kk > 0) ? 1u : 0u;
          const uint64_t bd = desc_sw128_kmajor(b + kk * 32);
          for (int m = 0; m < ntiles; ++m) {
            const uint64_t ad = desc_sw128_kmajor(a + m * C::A_BYTES + kk * 32);
            mma_ss(tmem + m * C::TCOLS, ad, bd, idesc, acc);
            if (BN > 256)
              mma_ss(tmem + m * C::TCOLS + 256, ad, desc_sw128_kmajor(b + 256 * 128 + kk * 32),
                     idesc2, acc);
          }
        }
      if (leader) tc_commit(&empty[s]);
      __syncwarp();
    }
    if (leader) {
      tc_commit(done);
      tc_commit(drain);
    }
    __syncwarp();
    for (uint32_t t = 0; t < (1u << 24) && !mbar_try(drain, 0); ++t) {
    }
  } else if (warp >= 2) {
    grid_dep_wait();  // the partial sums may still be read by the previous reduction
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    if (mbar_wait(done, 0, status, 503, abort, 256)) {
      tc_fence_after();
      for (int mi = 0; mi < ntiles; ++mi) {
        const int m = (mt0 + mi) * 128 + q * 32 + lane;
        float* out = part + ((size_t)split * Mtot + grp.prow[g] + m) * N + blockIdx.y * BN;
#pragma unroll
        for (int c0 = 0; c0 < BN; c0 += 16) {
          uint32_t v[16];
          tmem_ld16(tmem + mi * C::TCOLS + ((uint32_t)(q * 32) << 16) + c0, v);
          tmem_wait_ld();
          if (m < M && kc1 > kc0) {
#pragma unroll
            for (int j = 0; j < 16; ++j)
              if (blockIdx.y * BN + c0 + j < N) out[c0 + j] = __uint_as_float(v[j]);
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, C::MT * C::TCOLS);
  }
}

// Per group (rows prow .. prow + M of the partial sums):
// mode 0: out[m][n] (+)= sum_s part[s][m][n] for n < Hout; bias[m] (+)= sum_s part[s][m][Hout]
// mode 1: m = p*Hout + o: out[p][n][o] (+)= sum_s part[s][m][n]; bias[m] (+)= sum_s part[s][m][Hout]
struct TNOut {
  float* out[kMaxGroups];
  float* bias[kMaxGroups];
  int mode[kMaxGroups];
  int M[kMaxGroups];
  int prow[kMaxGroups];
  int n_groups;
};

__global__ void k_gemm_tn_reduce(const float* __restrict__ part, int splits, int Mtot, int N,
                                 int Hout, TNOut o, int accumulate) {
  grid_dep_wait();
  const int64_t total = (int64_t)Mtot * (Hout + 1);
  const size_t stride = (size_t)Mtot * N;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int mm = (int)(t / (Hout + 1)), n = (int)(t % (Hout + 1));
    int g = 0;
    while (g + 1 < o.n_groups && mm >= o.prow[g + 1]) ++g;
    const int m = mm - o.prow[g];
    if (m >= o.M[g]) continue;
    const float* src = part + (size_t)mm * N + n;
    // four independent partial sums keep several loads in flight; fixed order, so deterministic
    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
    int q = 0;
    for (; q + 4 <= splits; q += 4) {
      s0 += src[(size_t)q * stride];
      s1 += src[(size_t)(q + 1) * stride];
      s2 += src[(size_t)(q + 2) * stride];
      s3 += src[(size_t)(q + 3) * stride];
    }
    for (; q < splits; ++q) s0 += src[(size_t)q * stride];
    const float s = (s0 + s1) + (s2 + s3);
    float* dst;
    if (n == Hout) {
      if (!o.bias[g]) continue;
      dst = o.bias[g] + m;
    } else if (o.mode[g] == 0) {
      dst = o.out[g] + (size_t)m * Hout + n;
    } else {
      const int p = m / Hout, oo = m % Hout;
      dst = o.out[g] + ((size_t)p * Hout + n) * Hout + oo;
    }
    *dst = accumulate ? *dst + s : s;
  }
}

// ---------------------------------------------------------------------------------------------
// Batched TN GEMM: C[b][m][n] (+)= sum_k A[b][m][k] B[b][n][k] (+ bias[b][n]); one 128 x BN output
// tile per CTA, K streamed in 64-wide chunks through a 4-stage TMA ring.
// One 128 x BN output tile per CTA.  Two stages keep a CTA under half of the SM's shared memory
// (96 KB at BN = 256) and its accumulator at most 256 TMEM columns, so two CTAs share an SM and one's
// epilogue overlaps the other's loads and MMAs (with four stages, one CTA per SM ran its load,
// MMA and epilogue back to back).
constexpr int kStagesB = 2;
template <int BN>
struct BCfg {
  static constexpr int A_BYTES = 128 * 128;
  static constexpr int B_BYTES = BN * 128;
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr int SMEM = kStagesB * STAGE + 1024 + 1024;
  static constexpr int TCOLS = BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
  static_assert(2 * (SMEM + 1024) <= 233472 && 2 * TCOLS <= 512, "two CTAs per SM");
  static_assert(4 * 32 * 33 * 4 <= kStagesB * STAGE, "epilogue transpose buffers");
};

struct BatchArgs {
  int M, N, kchunks, a3d, b3d;
  float* C;
  int64_t ldc, sC;
  const float* bias;
  int64_t sBias;
  int accumulate;
  int vec;  // C rows (and bias) 16-byte aligned: each thread stores its row as float4
  // instead of C: the product rounded to bf16 and stored transposed, CT[n * ldT + m] (batch 1,
  // no bias, no accumulation; M even, N a multiple of 32, ldT even)
  __nv_bfloat16* CT;
  int64_t ldT;
};

template <int BN>
__global__ void __launch_bounds__(192, 2)
    k_gemm_bf16(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                BatchArgs g, int* status) {
  using C = BCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStagesB * C::STAGE);
  uint64_t* empty = full + kStagesB;
  uint64_t* done = empty + kStagesB;
  uint64_t* drain = done + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
  volatile int* abort = abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = blockIdx.x, nt = blockIdx.y, b = blockIdx.z;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStagesB; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(done, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TCOLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (warp == 0 && lane == 0) {
    uint32_t issued[kStagesB] = {};
    for (int kc = 0; kc < g.kchunks; ++kc) {
      const int s = kc % kStagesB;
      if (!mbar_wait(&empty[s], ((kc / kStagesB) & 1) ^ 1, status, 511, abort, 32)) break;
      ++issued[s];
      mbar_expect_tx(&full[s], C::STAGE);
      uint8_t* st = smem + s * C::STAGE;
      if (g.a3d) tma_load_3d(st, &tmA, &full[s], kc * 64, mt * 128, b);
      else tma_load_2d(st, &tmA, &full[s], kc * 64, mt * 128);
      if (g.b3d) tma_load_3d(st + C::A_BYTES, &tmB, &full[s], kc * 64, nt * BN, b);
      else tma_load_2d(st + C::A_BYTES, &tmB, &full[s], kc * 64, nt * BN);
    }
    if (*abort)
      for (int s = 0; s < kStagesB; ++s)
        for (uint32_t t = 0; issued[s] && t < (1u << 22) && !mbar_try(&full[s], (issued[s] - 1) & 1); ++t) {
        }
  } else if (warp == 1) {
    const bool leader = elect_one_sync();
    constexpr uint32_t idesc = idesc_bf16_f32(128, BN);
    for (int kc = 0; kc < g.kchunks; ++kc) {
      const int s = kc % kStagesB;
      if (!mbar_wait(&full[s], (kc / kStagesB) & 1, status, 512, abort)) break;
      tc_fence_after();
      const uint32_t a = smem_u32(smem + s * C::STAGE), bb = a + C::A_BYTES;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        if (leader)
          mma_ss(tmem, desc_sw128_kmajor(a + kk * 32), desc_sw128_kmajor(bb + kk * 32), idesc,
                 (kc > 0 || kk > 0) ? 1u : 0u);
      if (leader) tc_commit(&empty[s]);
      __syncwarp();
    }
    if (leader) {
      tc_commit(done);
      tc_commit(drain);
    }
    __syncwarp();
    for (uint32_t t = 0; t < (1u << 24) && !mbar_try(drain, 0); ++t) {
    }
  } else if (warp >= 2 && g.CT) {
    // thread = row m, 32 consecutive columns per round; a lane pair (rows m, m + 1) swaps its
    // packed column pairs so that each lane stores 4-byte words of two rows of one column
    const int q = warp & 3;
    if (mbar_wait(done, 0, status, 513, abort, 128)) {
      tc_fence_after();
      const int m = mt * 128 + q * 32 + lane;
      const bool odd = lane & 1;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        const int n0 = nt * BN + c0;
        if (n0 >= g.N) break;  // the same for the whole warp
        uint32_t v[32];
        tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + c0, v);
        tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + c0 + 16, v + 16);
        tmem_wait_ld();
        __nv_bfloat16* base = g.CT + (size_t)(n0 + odd) * g.ldT + (m & ~1);
        const bool live = (m & ~1) < g.M;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          __nv_bfloat162 h2 = __floats2bfloat162_rn(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
          const uint32_t pk = *reinterpret_cast<uint32_t*>(&h2);
          const uint32_t other = __shfl_xor_sync(0xffffffffu, pk, 1);
          const uint32_t word = odd ? __byte_perm(other, pk, 0x7632) : __byte_perm(pk, other, 0x5410);
          if (live) *reinterpret_cast<uint32_t*>(base + (size_t)(2 * j) * g.ldT) = word;
        }
      }
    }
  } else if (warp >= 2 && g.vec) {
    // each warp drains its 32 TMEM lanes (rows), 32 columns at a time: a thread holds 32
    // consecutive columns of its own row and writes them as 8 float4; the accumulating form reads
    // the 8 previous float4 first, all in flight at once
    const int q = warp & 3;
    if (mbar_wait(done, 0, status, 513, abort, 128)) {
      tc_fence_after();
      const float* brow = g.bias ? g.bias + (size_t)b * g.sBias : nullptr;
      float* cbase = g.C + (size_t)b * g.sC;
      const int m = mt * 128 + q * 32 + lane;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        const int n0 = nt * BN + c0;
        if (n0 >= g.N) break;  // the same for the whole warp
        uint32_t v[32];
        tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + c0, v);
        tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + c0 + 16, v + 16);
        tmem_wait_ld();
        if (m >= g.M) continue;
        float* dst = cbase + (size_t)m * g.ldc + n0;
        if (n0 + 32 <= g.N) {
          float4 prev[8];
          if (g.accumulate) {
#pragma unroll
            for (int j = 0; j < 8; ++j) prev[j] = reinterpret_cast<const float4*>(dst)[j];
          }
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            float4 o = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                   __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
            if (brow) {
              const float4 bv = reinterpret_cast<const float4*>(brow + n0)[j];
              o.x += bv.x; o.y += bv.y; o.z += bv.z; o.w += bv.w;
            }
            if (g.accumulate) { o.x += prev[j].x; o.y += prev[j].y; o.z += prev[j].z; o.w += prev[j].w; }
            reinterpret_cast<float4*>(dst)[j] = o;
          }
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (n0 + j < g.N) {
              const float x = __uint_as_float(v[j]) + (brow ? brow[n0 + j] : 0.f);
              dst[j] = g.accumulate ? dst[j] + x : x;
            }
        }
      }
    }
  } else if (warp >= 2) {
    // each warp drains its 32 TMEM lanes (rows) 32 columns at a time through a padded SMEM
    // transpose so that every global store instruction writes 32 consecutive columns of one row
    const int q = warp & 3;
    if (mbar_wait(done, 0, status, 513, abort, 128)) {
      tc_fence_after();
      float* sbuf = reinterpret_cast<float*>(smem) + (warp - 2) * 32 * 33;  // stages are idle now
      const float* brow = g.bias ? g.bias + (size_t)b * g.sBias : nullptr;
      float* cbase = g.C + (size_t)b * g.sC;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t v[32];
        tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + c0, v);
        tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + c0 + 16, v + 16);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 32; ++j) sbuf[lane * 33 + j] = __uint_as_float(v[j]);
        __syncwarp();
        const int n = nt * BN + c0 + lane;
        const float bv = (brow && n < g.N) ? brow[n] : 0.f;
#pragma unroll 4
        for (int rr = 0; rr < 32; ++rr) {
          const int m = mt * 128 + q * 32 + rr;
          if (m < g.M && n < g.N) {
            float* dst = cbase + (size_t)m * g.ldc + n;
            const float x = sbuf[rr * 33 + lane] + bv;
            *dst = g.accumulate ? *dst + x : x;
          }
        }
        __syncwarp();
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, C::TCOLS);
  }
}

}  // namespace

namespace {
cudaError_t gemm_bf16_tn_any(const void* A, int64_t lda, int64_t sA, const void* B, int64_t ldb,
                             int64_t sB, int M, int N, int K, int batch, float* Cout, int64_t ldc,
                             int64_t sC, const float* bias, int64_t sBias, int accumulate,
                             __nv_bfloat16* CT, int64_t ldT, int* status, cudaStream_t st) {
  if (M <= 0 || N <= 0 || batch <= 0) return cudaSuccess;
  if (K <= 0 || (lda % 8) || (ldb % 8) || (sA % 8) || (sB % 8)) return cudaErrorInvalidValue;
  const int BN = N <= 64 ? 64 : N <= 128 ? 128 : N <= 192 ? 192 : 256;
  CUtensorMap ta, tb;
  const bool a3 = batch > 1 && sA != 0, b3 = batch > 1 && sB != 0;
  if (!(a3 ? make_map_3d(&ta, A, batch, M, K, lda, sA, 128) : make_map_ld(&ta, A, M, K, lda, 128)) ||
      !(b3 ? make_map_3d(&tb, B, batch, N, K, ldb, sB, BN) : make_map_ld(&tb, B, N, K, ldb, BN)))
    return cudaErrorInvalidValue;
  const int vec = (reinterpret_cast<uintptr_t>(Cout) % 16 == 0) && ldc % 4 == 0 && sC % 4 == 0 &&
                  (!bias || (reinterpret_cast<uintptr_t>(bias) % 16 == 0 && sBias % 4 == 0));
  BatchArgs g{M, N, (K + 63) / 64, a3 ? 1 : 0, b3 ? 1 : 0, Cout, ldc, sC, bias, sBias, accumulate,
              vec, CT, ldT};
  dim3 grid((M + 127) / 128, (N + BN - 1) / BN, batch);
  cudaError_t e;
#define BG_GEMM16_CASE(BNV)                                                                    \
  e = cudaFuncSetAttribute(k_gemm_bf16<BNV>, cudaFuncAttributeMaxDynamicSharedMemorySize,      \
                           BCfg<BNV>::SMEM);                                                   \
  if (e != cudaSuccess) return e;                                                              \
  k_gemm_bf16<BNV><<<grid, 192, BCfg<BNV>::SMEM, st>>>(ta, tb, g, status);
  switch (BN) {
    case 64: BG_GEMM16_CASE(64) break;
    case 128: BG_GEMM16_CASE(128) break;
    case 192: BG_GEMM16_CASE(192) break;
    default: BG_GEMM16_CASE(256) break;
  }
#undef BG_GEMM16_CASE
  note_launch();
  return cudaGetLastError();
}
}  // namespace

cudaError_t gemm_bf16_tn(const void* A, int64_t lda, int64_t sA, const void* B, int64_t ldb,
                         int64_t sB, int M, int N, int K, int batch, float* Cout, int64_t ldc,
                         int64_t sC, const float* bias, int64_t sBias, int accumulate, int* status,
                         cudaStream_t st) {
  return gemm_bf16_tn_any(A, lda, sA, B, ldb, sB, M, N, K, batch, Cout, ldc, sC, bias, sBias,
                          accumulate, nullptr, 0, status, st);
}

cudaError_t gemm_bf16_tn_outT(const void* A, int64_t lda, const void* B, int64_t ldb, int M, int N,
                              int K, __nv_bfloat16* CT, int64_t ldT, int* status, cudaStream_t st) {
  if (!CT || (M % 2) || (N % 32) || (ldT % 2) || ldT < M ||
      (reinterpret_cast<uintptr_t>(CT) % 4))
    return cudaErrorInvalidValue;
  return gemm_bf16_tn_any(A, lda, 0, B, ldb, 0, M, N, K, 1, nullptr, 0, 0, nullptr, 0, 0, CT, ldT,
                          status, st);
}

size_t gemm_tn_part_floats(int M, int N, int64_t K) {
  const int64_t kchunks = (K + 63) / 64;
  const int mt = (M + 127) / 128;
  const int64_t splits = std::max<int64_t>(1, std::min<int64_t>(kchunks, (512 + mt - 1) / mt));
  return (size_t)splits * M * N;
}

cudaError_t gemm_tn_multi(const TNProblem* pr, int n, int Hout, int64_t K, int accumulate,
                          float* part, size_t part_floats, int* status, cudaStream_t st) {
  const int N = Hout + 16;  // Hout gradient columns, one ones-column (bias), padding to 16
  if (N != 48 && N != 80 && N != 144 && N != 272) return cudaErrorInvalidValue;
  if (n < 1 || n > kMaxGroups) return cudaErrorInvalidValue;
  const int64_t kchunks = (K + 63) / 64;
  TNGroups grp{};
  TNOut o{};
  const int MT = N <= 256 ? 2 : 1;  // M tiles per CTA (GCfg::MT)
  int mt = 0, Mtot = 0;
  for (int g = 0; g < n; ++g) {
    if (!make_map_ld(&grp.a[g], pr[g].A, pr[g].M, K, pr[g].lda, 128) ||
        !make_map_ld(&grp.b[g], pr[g].B, N - 16, K, pr[g].ldb, N - 16))
      return cudaErrorInvalidValue;
    mt += ((pr[g].M + 127) / 128 + MT - 1) / MT;
    grp.it_end[g] = mt;
    grp.M[g] = o.M[g] = pr[g].M;
    grp.prow[g] = o.prow[g] = Mtot;
    o.out[g] = pr[g].out;
    o.bias[g] = pr[g].bias;
    o.mode[g] = pr[g].mode;
    Mtot += pr[g].M;
  }
  for (int g = n; g < kMaxGroups; ++g) grp.it_end[g] = mt;
  o.n_groups = n;
  const int sms = gemm_tn_num_sms();
  // at most one CTA per SM, so that all of them run in one wave (a partial second wave of even a
  // few CTAs would nearly double the time of this HBM-bound pass)
  int splits = (int)std::max<int64_t>(1, std::min<int64_t>(kchunks, std::max(1, sms / mt)));
  while (splits > 1 && (size_t)splits * Mtot * N > part_floats) --splits;
  // the kernel writes its partial sums even when it does not split K
  if ((size_t)splits * Mtot * N > part_floats) return cudaErrorInvalidValue;
  const int per = (int)((kchunks + splits - 1) / splits);
  splits = (int)((kchunks + per - 1) / per);
  dim3 grid(mt, 1, splits);
  cudaError_t e;
#define BG_GEMM_CASE(BNV)                                                                      \
  e = cudaFuncSetAttribute(k_gemm_tn<BNV>, cudaFuncAttributeMaxDynamicSharedMemorySize,        \
                           GCfg<BNV>::SMEM);                                                   \
  if (e != cudaSuccess) return e;                                                              \
  e = launch_pdl(k_gemm_tn<BNV>, grid, dim3(192), GCfg<BNV>::SMEM, st, grp, part, Mtot, N,        \
                 (int)kchunks, per, status);                                                   \
  if (e != cudaSuccess) return e;
  if (N == 48) {
    BG_GEMM_CASE(48)
  } else if (N == 80) {
    BG_GEMM_CASE(80)
  } else if (N == 144) {
    BG_GEMM_CASE(144)
  } else {
    BG_GEMM_CASE(272)
  }
#undef BG_GEMM_CASE
  note_launch();
  const int64_t total = (int64_t)Mtot * (Hout + 1);
  e = launch_pdl(k_gemm_tn_reduce, dim3((unsigned)std::min<int64_t>((total + 255) / 256, 4096)),
                 dim3(256), 0, st, (const float*)part, splits, Mtot, N, Hout, o, accumulate);
  note_launch();
  return e;
}

namespace {
// One warp waits, through the same bounded wait as every pipeline role, on an mbarrier that
// nothing arrives on: after the poll cap it records a timeout (site 901) in the status word and
// returns, as a stalled kernel would.
__global__ void k_wait_selftest(int* status) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  volatile int* abort = &abort_flag;
  if (threadIdx.x == 0) mbar_wait(&bar, 0, status, 901, abort, 64);
  __syncthreads();
}
}  // namespace

cudaError_t wait_selftest(int* status, cudaStream_t st) {
  k_wait_selftest<<<1, 32, 0, st>>>(status);
  note_launch();
  return cudaGetLastError();
}

cudaError_t gemm_tn(const void* A, int64_t lda, const void* B, int64_t ldb, int M, int Hout,
                    int64_t K, int mode, float* out, float* bias, int accumulate, float* part,
                    size_t part_floats, int* status, cudaStream_t st) {
  const TNProblem pr{A, lda, B, ldb, M, mode, out, bias};
  return gemm_tn_multi(&pr, 1, Hout, K, accumulate, part, part_floats, status, st);
}

}  // namespace bg

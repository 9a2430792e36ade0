// GRU cell (Cho et al.; named in Section 2 and Algorithm 1) forward and backward on tcgen05.
// Gate convention: rows r, z, n of W_ih / W_hh;
//   r = sigma(Wi_r x + b_ir + Wh_r h + b_hr),  z = sigma(Wi_z x + b_iz + Wh_z h + b_hz),
//   n = tanh(Wi_n x + b_in + r (Wh_n h + b_hn)),  h' = (1 - z) n + z h,
// with x the summed messages Y and h the state E; padding rows stay 0.
//
// Pre-activations live in TMEM: [r|z] = Y Wi_rz^T + E Wh_rz^T (2H columns: both products
// accumulate into one tile), Wi_n x (H) and Wh_n h (H).  The forward epilogue applies the gates
// and writes E(t+1) row-major and transposed (the next band product's operand).  The backward
// recomputes the same products, forms the gate gradients in registers, writes them back into the
// TMEM columns it has just read as the bf16 A operand of dX = dgi W_ih and dH = dgh W_hh (chained
// MMAs that accumulate into the freed Wi_n x / Wh_n h columns), and stores dX^T (the
// transposed-band operand), the running state gradient and dgi^T, dgh^T for the weight gradients.
//
// Both kernels are persistent (one CTA per SM) and warp-specialised: warp 0 streams 128-row
// tiles of Y and E through a two-stage TMA ring (the weights stay resident), warp 1 issues the
// MMAs into two TMEM accumulator sets, and four epilogue warpgroups (one per 16 state columns,
// eight at a time) drain them, so loads and MMAs of tile i+1 overlap the epilogue of tile i.
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>

#include "gemm_tc.h"
#include "gru_tc.h"
#include "kernels.h"
#include "tc_util.cuh"

namespace bg {

using namespace tc;

namespace {

// The kernels below take H = KH in {32, 64}: the state fits one 64-column (128-byte) swizzle atom
// of the tile, whose columns KH .. 63 the tensor maps fill with zeros at KH = 32, and only the
// first KH / 16 K steps are issued.
constexpr int kEpiWarps = 16; // four epilogue warpgroups of up to 16 state columns each
constexpr int kThreads = 128 + 32 * kEpiWarps;  // warp 0 TMA, warp 1 MMA, warps 4-19 epilogue
template <int KH>
__host__ __device__ constexpr int epi_warps() { return 4 * (KH / 16); }  // warps with columns

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t* r) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
                 "=r"(r[6]), "=r"(r[7])
               : "r"(taddr));
}

__device__ __forceinline__ void tmem_st4(uint32_t taddr, const uint32_t* r) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1,%2,%3,%4};" ::"r"(taddr), "r"(r[0]),
               "r"(r[1]), "r"(r[2]), "r"(r[3])
               : "memory");
}

// One arrive per warp once every lane of it is done.
__device__ __forceinline__ void warp_arrive(uint64_t* bar) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}

__device__ __forceinline__ uint32_t pk2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// tanh on the special-function unit (tanh.approx.f32: relative error about 2^-11, below the bf16
// rounding of the state) and the logistic function through sigma(x) = (1 + tanh(x / 2)) / 2
__device__ __forceinline__ float tanh_fast(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float sigm(float x) { return fmaf(0.5f, tanh_fast(0.5f * x), 0.5f); }

// Gate biases in shared memory as four H-vectors: b_ir + b_hr, b_iz + b_hz, b_in, b_hn (the r and z
// biases enter only as sums); a thread reads those of its four columns c .. c+3 as one float4 each.
struct GateBias {
  float4 r, z, in, hn;
};
__device__ __forceinline__ GateBias gate_bias(const float* b, int H, int c) {
  GateBias g;
  g.r = *reinterpret_cast<const float4*>(b + c);
  g.z = *reinterpret_cast<const float4*>(b + H + c);
  g.in = *reinterpret_cast<const float4*>(b + 2 * H + c);
  g.hn = *reinterpret_cast<const float4*>(b + 3 * H + c);
  return g;
}
__device__ __forceinline__ float f4(const float4& v, int u) {
  return u == 0 ? v.x : u == 1 ? v.y : u == 2 ? v.z : v.w;
}
__device__ __forceinline__ void fill_gate_bias(float* bias, const float* b_ih, const float* b_hh,
                                               int H) {
  for (int t = threadIdx.x; t < H; t += blockDim.x) {
    bias[t] = b_ih[t] + b_hh[t];
    bias[H + t] = b_ih[H + t] + b_hh[H + t];
    bias[2 * H + t] = b_ih[2 * H + t];
    bias[3 * H + t] = b_hh[2 * H + t];
  }
}

// 8 consecutive bf16 of row r (columns c0 .. c0+7, c0 % 8 == 0): one swizzled 16-byte chunk.
__device__ __forceinline__ void read_sw128_row8(const uint8_t* tile, int r, int c0, float* out) {
  const uint8_t* row = tile + (c0 / 64) * 128 * 128 + r * 128;
  const uint4 v = *reinterpret_cast<const uint4*>(row + ((((c0 % 64) / 8) ^ (r & 7)) << 4));
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    out[2 * e] = __uint_as_float(w[e] << 16);
    out[2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
  }
}

// 8 consecutive fp32 of row r (columns c0 .. c0+7, c0 % 8 == 0) of a 128-row tile stored as
// 32-column boxes (128-byte rows) with the 128-byte swizzle.
__device__ __forceinline__ void read_sw128_f32_row8(const uint8_t* tile, int r, int c0, float4* out) {
  const uint8_t* row = tile + (c0 / 32) * 128 * 128 + r * 128;
  const int j0 = (c0 % 32) / 4;
  out[0] = *reinterpret_cast<const float4*>(row + (((j0) ^ (r & 7)) << 4));
  out[1] = *reinterpret_cast<const float4*>(row + (((j0 + 1) ^ (r & 7)) << 4));
}

// N bf16 pairs (columns h0 + 2j, h0 + 2j + 1 of this lane's row) stored transposed,
// dst[(h0 + 2j + u) * ld + row], as 4-byte words of two rows: the rows of a warp are consecutive
// (row parity = lane parity), so a lane pair swaps its pairs with one shuffle and the even lane
// writes column h0 + 2j of both rows, the odd lane column h0 + 2j + 1.  Every lane of the warp
// calls it; ld and the row pair's first row are even.
template <int N>
__device__ __forceinline__ void store_T_pairs(__nv_bfloat16* dst, int64_t ld, int row, int h0,
                                              const uint32_t* pk) {
  const int odd = row & 1;
  __nv_bfloat16* base = dst + (size_t)(h0 + odd) * ld + (row & ~1);
#pragma unroll
  for (int j = 0; j < N; ++j) {
    const uint32_t other = __shfl_xor_sync(0xffffffffu, pk[j], 1);
    const uint32_t word = odd ? __byte_perm(other, pk[j], 0x7632) : __byte_perm(pk[j], other, 0x5410);
    *reinterpret_cast<uint32_t*>(base + (size_t)(2 * j) * ld) = word;
  }
}
__device__ __forceinline__ void store_T4(__nv_bfloat16* dst, int64_t ld, int row, int h0,
                                         const uint32_t* pk) {
  store_T_pairs<4>(dst, ld, row, h0, pk);
}
__device__ __forceinline__ void store_T8(__nv_bfloat16* dst, int64_t ld, int row, int h0,
                                         const uint32_t* pk) {
  store_T_pairs<8>(dst, ld, row, h0, pk);
}

template <int KH>
struct GruSmem {
  static constexpr int TILE = 128 * 128;  // 128 rows x 64 bf16 (columns >= KH zero)
  static constexpr int G = 128 * KH * 4;  // 128 rows x KH fp32 (incoming state gradient, backward)
  static constexpr int W = 3 * KH * 128;  // [3H][64] bf16 (also [H][3H] as 64-column atoms)
  static constexpr int WT_ATOMS = (3 * KH + 63) / 64;
  static constexpr int FWD_T = 2 * W;     // tile ring after W_ih, W_hh
  static constexpr int BWD_T = 4 * W;     // tile ring after W_ih, W_hh, W_ih^T, W_hh^T
  static constexpr int FWD_STAGE = 2 * TILE;      // Y, E
  static constexpr int BWD_STAGE = 2 * TILE + G;  // Y, E, g
  // dynamic shared memory: the ring plus 1 KB of slack for aligning its base to 1024 bytes; the
  // barriers and biases are static (< 2 KB) and count toward the same 227 KB per block
  static constexpr int FWD = FWD_T + 2 * FWD_STAGE + 1024;
  static constexpr int BWD = BWD_T + 2 * BWD_STAGE + 1024;
  static_assert(BWD + 2048 <= 232448, "shared memory");
  static_assert(WT_ATOMS * KH * 128 <= W, "transposed weights");
};

struct GruBars {
  uint64_t w_full, t_full[2], t_empty[2], acc_full[2], acc_empty[2], ops_ready[2], ph2_full[2];
  uint64_t drain;
  uint32_t tmem_slot;
  int abort;
};

// Issues [r|z], Wi_n x, Wh_n h for one tile into the accumulator set at `acc` (K = H).
template <int KH>
__device__ __forceinline__ void gru_gate_mmas(uint32_t acc, uint32_t sY, uint32_t sE, uint32_t sWih,
                                              uint32_t sWhh) {
  constexpr uint32_t id_rz = idesc_bf16_f32(128, 2 * KH), id_h = idesc_bf16_f32(128, KH);
#pragma unroll
  for (int kk = 0; kk < KH / 16; ++kk) {
    const uint64_t aY = desc_sw128_kmajor(sY + kk * 32), aE = desc_sw128_kmajor(sE + kk * 32);
    mma_ss(acc + 0, aY, desc_sw128_kmajor(sWih + kk * 32), id_rz, kk > 0);
    mma_ss(acc + 0, aE, desc_sw128_kmajor(sWhh + kk * 32), id_rz, 1u);
    mma_ss(acc + 2 * KH, aY, desc_sw128_kmajor(sWih + 2 * KH * 128 + kk * 32), id_h, kk > 0);
    mma_ss(acc + 3 * KH, aE, desc_sw128_kmajor(sWhh + 2 * KH * 128 + kk * 32), id_h, kk > 0);
  }
}

// Common prologue: barrier init, bias copy, TMEM allocation (512 columns: two accumulator sets).
template <int KH>
__device__ __forceinline__ void gru_setup(GruBars* b, float* bias, const float* b_ih,
                                          const float* b_hh, int warp) {
  fill_gate_bias(bias, b_ih, b_hh, KH);
  if (threadIdx.x == 0) {
    mbar_init(&b->w_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&b->t_full[i], 1);
      mbar_init(&b->t_empty[i], epi_warps<KH>());
      mbar_init(&b->acc_full[i], 1);
      mbar_init(&b->acc_empty[i], epi_warps<KH>());
      mbar_init(&b->ops_ready[i], epi_warps<KH>());
      mbar_init(&b->ph2_full[i], 1);
    }
    mbar_init(&b->drain, 1);
    b->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&b->tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // TMEM is held: the next kernel in the stream may be scheduled on SMs as they free up
  grid_dep_launch();
}

// Tile producer shared by both kernels: two-stage ring of (Y, E) tiles and, backward, the fp32
// incoming gradient tile (KH / 32 boxes of 32 columns with the 128-byte swizzle).
template <int KH>
__device__ __forceinline__ void gru_produce_tiles(GruBars* b, uint8_t* ring, int stage,
                                                  const CUtensorMap* tY, const CUtensorMap* tE,
                                                  const CUtensorMap* tG, int n_tiles, int* status,
                                                  volatile int* abort) {
  // the tiles are the previous kernel's output (the weights, loaded before this, are not)
  grid_dep_wait();
  uint32_t issued[2] = {0, 0};
  int i = 0;
  for (int t = blockIdx.x; t < n_tiles && !*abort; t += gridDim.x, ++i) {
    const int s = i & 1;
    if (!mbar_wait(&b->t_empty[s], ((i >> 1) & 1) ^ 1, status, 611, abort, 64)) break;
    ++issued[s];
    uint8_t* st = ring + s * stage;
    using SM = GruSmem<KH>;
    mbar_expect_tx(&b->t_full[s], 2 * SM::TILE + (tG ? SM::G : 0));
    tma_load_2d(st, tY, &b->t_full[s], 0, t * 128);
    tma_load_2d(st + SM::TILE, tE, &b->t_full[s], 0, t * 128);
    if (tG)
      for (int a = 0; a < KH / 32; ++a)
        tma_load_2d(st + 2 * SM::TILE + a * 128 * 128, tG, &b->t_full[s], 32 * a, t * 128);
  }
  if (*abort)
    for (int s = 0; s < 2; ++s)
      for (uint32_t k = 0; issued[s] && k < (1u << 22) && !mbar_try(&b->t_full[s], (issued[s] - 1) & 1); ++k) {
      }
}

template <int KH>
__global__ void __launch_bounds__(kThreads, 1)
    k_gru_fwd_tc(const __grid_constant__ CUtensorMap tY, const __grid_constant__ CUtensorMap tE,
                 const __grid_constant__ CUtensorMap tWih, const __grid_constant__ CUtensorMap tWhh,
                 const float* __restrict__ b_ih, const float* __restrict__ b_hh,
                 __nv_bfloat16* __restrict__ En, __nv_bfloat16* __restrict__ EnT, int64_t ld_T,
                 int n_tiles, int n_real, int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  __shared__ GruBars bars;
  __shared__ __align__(16) float bias[4 * KH];
  using SM = GruSmem<KH>;
  constexpr int kAcc = 4 * KH;  // TMEM columns per accumulator set
  volatile int* abort = &bars.abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  gru_setup<KH>(&bars, bias, b_ih, b_hh, warp);
  const uint32_t tmem = bars.tmem_slot;
  uint8_t* ring = smem + SM::FWD_T;

  if (warp == 0 && lane == 0) {
    mbar_expect_tx(&bars.w_full, 2 * SM::W);
    tma_load_2d(smem, &tWih, &bars.w_full, 0, 0);
    tma_load_2d(smem + SM::W, &tWhh, &bars.w_full, 0, 0);
    gru_produce_tiles<KH>(&bars, ring, SM::FWD_STAGE, &tY, &tE, nullptr, n_tiles, status, abort);
    if (*abort)
      for (uint32_t k = 0; k < (1u << 22) && !mbar_try(&bars.w_full, 0); ++k) {
      }
  } else if (warp == 1) {
    const bool leader = elect_one_sync();
    if (mbar_wait(&bars.w_full, 0, status, 612, abort)) {
      int i = 0;
      for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++i) {
        const int s = i & 1, a = i & 1;
        if (!mbar_wait(&bars.t_full[s], (i >> 1) & 1, status, 613, abort)) break;
        if (!mbar_wait(&bars.acc_empty[a], ((i >> 1) & 1) ^ 1, status, 614, abort)) break;
        tc_fence_after();
        const uint32_t sY = smem_u32(ring + s * 2 * SM::TILE);
        if (leader) {
          gru_gate_mmas<KH>(tmem + a * kAcc, sY, sY + SM::TILE, smem_u32(smem),
                        smem_u32(smem + SM::W));
          tc_commit(&bars.acc_full[a]);
        }
        __syncwarp();
      }
    }
    if (leader) tc_commit(&bars.drain);
    __syncwarp();
    for (uint32_t k = 0; k < (1u << 24) && !mbar_try(&bars.drain, 0); ++k) {
    }
  } else if (warp >= 4 && (warp - 4) / 4 < KH / 16) {
    grid_dep_wait();  // outputs may still be in use by the previous kernel
    const int g = (warp - 4) / 4, h0 = 16 * g;
    const int r = (warp & 3) * 32 + lane;
    const uint32_t lb = (uint32_t)((warp & 3) * 32) << 16;
    int i = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++i) {
      const int s = i & 1, a = i & 1;
      if (!mbar_wait(&bars.acc_full[a], (i >> 1) & 1, status, 615, abort, 64)) break;
      tc_fence_after();
      const uint32_t acc = tmem + lb + a * kAcc;
      const uint8_t* etile = ring + s * 2 * SM::TILE + SM::TILE;
      const int row = t * 128 + r;
      const bool real = row < n_real;
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int hs = h0 + 8 * hh;
        uint32_t vr[8], vz[8], vn[8], vh[8];
        tmem_ld8(acc + hs, vr);
        tmem_ld8(acc + KH + hs, vz);
        tmem_ld8(acc + 2 * KH + hs, vn);
        tmem_ld8(acc + 3 * KH + hs, vh);
        tmem_wait_ld();
        float e[8];
        read_sw128_row8(etile, r, hs, e);
        if (hh == 1) {
          // accumulators and the state tile of this tile are no longer needed
          tc_fence_before();
          warp_arrive(&bars.acc_empty[a]);
          warp_arrive(&bars.t_empty[s]);
        }
        uint32_t pk[4];
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          const GateBias gb = gate_bias(bias, KH, hs + 4 * q);
          float o[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int j = 4 * q + u;
            const float rr = sigm(__uint_as_float(vr[j]) + f4(gb.r, u));
            const float zz = sigm(__uint_as_float(vz[j]) + f4(gb.z, u));
            const float nn = tanh_fast(__uint_as_float(vn[j]) + f4(gb.in, u) +
                                       rr * (__uint_as_float(vh[j]) + f4(gb.hn, u)));
            o[u] = real ? (1.f - zz) * nn + zz * e[j] : 0.f;
          }
          pk[2 * q] = pk2(o[0], o[1]);
          pk[2 * q + 1] = pk2(o[2], o[3]);
        }
        *reinterpret_cast<uint4*>(En + (size_t)row * KH + hs) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        if (EnT) store_T4(EnT, ld_T, row, hs, pk);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// A-operand column (relative to an accumulator set) of gate-gradient K step kk (16 values of one
// gate) after the in-place rewrite.  Columns h in [32c + 16sb, +16) of chunk c, sub-chunk sb, are
// read and then overwritten as: r window [32c + 16sb, +16) = (dgi_r | dgi_z) pairs, z window
// [H + 32c + 16sb, +16) = (dgi_n | dgh_n) pairs; dgh_r = dgi_r and dgh_z = dgi_z.
template <int KH>
__device__ __forceinline__ uint32_t dg_col(int kk, bool hidden) {
  const int gate = kk / (KH / 16), hh = (kk % (KH / 16)) * 16, c = hh / 32, sb = (hh % 32) / 16;
  const int base = c * 32 + sb * 16;
  if (gate == 0) return base;
  if (gate == 1) return base + 8;
  return KH + base + (hidden ? 8 : 0);
}

template <int KH>
__global__ void __launch_bounds__(kThreads, 1)
    k_gru_bwd_tc(const __grid_constant__ CUtensorMap tY, const __grid_constant__ CUtensorMap tE,
                 const __grid_constant__ CUtensorMap tWih, const __grid_constant__ CUtensorMap tWhh,
                 const __grid_constant__ CUtensorMap tWihT, const __grid_constant__ CUtensorMap tWhhT,
                 const __grid_constant__ CUtensorMap tG,
                 const float* __restrict__ b_ih, const float* __restrict__ b_hh,
                 float* __restrict__ gout,
                 __nv_bfloat16* __restrict__ dXT, int64_t ld_x, __nv_bfloat16* __restrict__ dgiT,
                 __nv_bfloat16* __restrict__ dhnT, int64_t ld_g, int n_tiles, int n_real,
                 int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  __shared__ GruBars bars;
  __shared__ __align__(16) float bias[4 * KH];
  using SM = GruSmem<KH>;
  constexpr int kAcc = 4 * KH;  // TMEM columns per accumulator set
  volatile int* abort = &bars.abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  gru_setup<KH>(&bars, bias, b_ih, b_hh, warp);
  const uint32_t tmem = bars.tmem_slot;
  uint8_t* ring = smem + SM::BWD_T;

  if (warp == 0 && lane == 0) {
    mbar_expect_tx(&bars.w_full, 2 * SM::W + 2 * SM::WT_ATOMS * KH * 128);
    tma_load_2d(smem, &tWih, &bars.w_full, 0, 0);
    tma_load_2d(smem + SM::W, &tWhh, &bars.w_full, 0, 0);
    for (int a = 0; a < SM::WT_ATOMS; ++a) {
      tma_load_2d(smem + 2 * SM::W + a * KH * 128, &tWihT, &bars.w_full, a * 64, 0);
      tma_load_2d(smem + 3 * SM::W + a * KH * 128, &tWhhT, &bars.w_full, a * 64, 0);
    }
    gru_produce_tiles<KH>(&bars, ring, SM::BWD_STAGE, &tY, &tE, &tG, n_tiles, status, abort);
    if (*abort)
      for (uint32_t k = 0; k < (1u << 22) && !mbar_try(&bars.w_full, 0); ++k) {
      }
  } else if (warp == 1) {
    const bool leader = elect_one_sync();
    constexpr uint32_t id_h = idesc_bf16_f32(128, KH);
    const uint32_t sIT = smem_u32(smem + 2 * SM::W), sHT = smem_u32(smem + 3 * SM::W);
    // dX = dgi W_ih, dH = dgh W_hh for tile j (accumulating into the freed n columns)
    auto phase2 = [&](int j) -> bool {
      const int a = j & 1;
      if (!mbar_wait(&bars.ops_ready[a], (j >> 1) & 1, status, 621, abort)) return false;
      tc_fence_after();
      if (leader) {
        const uint32_t acc = tmem + a * kAcc;
#pragma unroll
        // K index 16 kk = gate * H + h of W^T: atom kk / 4, 32-byte step kk % 4
        for (int kk = 0; kk < 3 * KH / 16; ++kk) {
          const uint32_t boff = (kk / 4) * KH * 128 + (kk % 4) * 32;
          mma_ts(acc + 2 * KH, acc + dg_col<KH>(kk, false), desc_sw128_kmajor(sIT + boff), id_h,
                 kk > 0);
          mma_ts(acc + 3 * KH, acc + dg_col<KH>(kk, true), desc_sw128_kmajor(sHT + boff), id_h,
                 kk > 0);
        }
        tc_commit(&bars.ph2_full[a]);
      }
      __syncwarp();
      return true;
    };
    if (mbar_wait(&bars.w_full, 0, status, 622, abort)) {
      int i = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++i) {
        const int s = i & 1, a = i & 1;
        if (!mbar_wait(&bars.t_full[s], (i >> 1) & 1, status, 623, abort)) break;
        if (!mbar_wait(&bars.acc_empty[a], ((i >> 1) & 1) ^ 1, status, 624, abort)) break;
        tc_fence_after();
        const uint32_t sY = smem_u32(ring + s * SM::BWD_STAGE);
        if (leader) {
          gru_gate_mmas<KH>(tmem + a * kAcc, sY, sY + SM::TILE, smem_u32(smem),
                        smem_u32(smem + SM::W));
          tc_commit(&bars.acc_full[a]);
        }
        __syncwarp();
        if (i >= 1) ok = phase2(i - 1);
      }
      if (ok && i >= 1) phase2(i - 1);
    }
    if (leader) tc_commit(&bars.drain);
    __syncwarp();
    for (uint32_t k = 0; k < (1u << 24) && !mbar_try(&bars.drain, 0); ++k) {
    }
  } else if (warp >= 4 && (warp - 4) / 4 < KH / 16) {
    grid_dep_wait();  // outputs may still be in use by the previous kernel
    const int g = (warp - 4) / 4, h0 = 16 * g;
    const int r = (warp & 3) * 32 + lane;
    const uint32_t lb = (uint32_t)((warp & 3) * 32) << 16;
    int i = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++i) {
      const int s = i & 1, a = i & 1;
      const int row = t * 128 + r;
      const bool real = row < n_real;
      if (!mbar_wait(&bars.acc_full[a], (i >> 1) & 1, status, 625, abort, 64)) break;
      tc_fence_after();
      const uint32_t acc = tmem + lb + a * kAcc;
      const uint8_t* etile = ring + s * SM::BWD_STAGE + SM::TILE;
      const uint8_t* gtile = etile + SM::TILE;
      float dhd[16];
      // packed gate gradients of both halves: the in-place rewrite below overwrites columns that
      // the second half still reads, so it waits until both halves are in registers
      uint32_t p_r[8], p_z[8], p_n[8], p_hn[8];
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        // columns hs .. hs+7: pairs 4hh .. 4hh+3 of this warpgroup's 16-column window h0
        const int hs = h0 + 8 * hh;
        uint32_t vr[8], vz[8], vn[8], vh[8];
        tmem_ld8(acc + hs, vr);
        tmem_ld8(acc + KH + hs, vz);
        tmem_ld8(acc + 2 * KH + hs, vn);
        tmem_ld8(acc + 3 * KH + hs, vh);
        tmem_wait_ld();
        float e[8];
        read_sw128_row8(etile, r, hs, e);
        float4 g4[2];
        read_sw128_f32_row8(gtile, r, hs, g4);
        if (hh == 1) warp_arrive(&bars.t_empty[s]);
        const int o = 4 * hh;
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          const float4 gv = g4[q];
          const float gg[4] = {gv.x, gv.y, gv.z, gv.w};
          const GateBias gb = gate_bias(bias, KH, hs + 4 * q);
          float dr[4], dz[4], dn[4], dhn[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int j = 4 * q + u;
            const float rr = sigm(__uint_as_float(vr[j]) + f4(gb.r, u));
            const float zz = sigm(__uint_as_float(vz[j]) + f4(gb.z, u));
            const float ghn = __uint_as_float(vh[j]) + f4(gb.hn, u);
            const float nn = tanh_fast(__uint_as_float(vn[j]) + f4(gb.in, u) + rr * ghn);
            const float gr = real ? gg[u] : 0.f;
            const float an = gr * (1.f - zz) * (1.f - nn * nn);
            dn[u] = an;
            dhn[u] = an * rr;
            dr[u] = an * ghn * rr * (1.f - rr);
            dz[u] = gr * (e[j] - nn) * zz * (1.f - zz);
            dhd[8 * hh + j] = gr * zz;
          }
          p_r[o + 2 * q] = pk2(dr[0], dr[1]); p_r[o + 2 * q + 1] = pk2(dr[2], dr[3]);
          p_z[o + 2 * q] = pk2(dz[0], dz[1]); p_z[o + 2 * q + 1] = pk2(dz[2], dz[3]);
          p_n[o + 2 * q] = pk2(dn[0], dn[1]); p_n[o + 2 * q + 1] = pk2(dn[2], dn[3]);
          p_hn[o + 2 * q] = pk2(dhn[0], dhn[1]); p_hn[o + 2 * q + 1] = pk2(dhn[2], dhn[3]);
        }
        // gate gradients transposed for the weight-gradient GEMM: dgi rows o = gate*H + h, and
        // of dgh only the n rows (its r and z rows equal dgi's)
        store_T4(dgiT, ld_g, row, hs, p_r + o);
        store_T4(dgiT + (size_t)KH * ld_g, ld_g, row, hs, p_z + o);
        store_T4(dgiT + (size_t)2 * KH * ld_g, ld_g, row, hs, p_n + o);
        store_T4(dhnT, ld_g, row, hs, p_hn + o);
      }
      // in-place rewrite into the columns just read (see dg_col): within the 16-column window h0,
      // r holds the 8 (dgi_r) pair columns then the 8 (dgi_z) ones, z the (dgi_n) then (dgh_n)
      tmem_st4(acc + h0, p_r);
      tmem_st4(acc + h0 + 4, p_r + 4);
      tmem_st4(acc + h0 + 8, p_z);
      tmem_st4(acc + h0 + 12, p_z + 4);
      tmem_st4(acc + KH + h0, p_n);
      tmem_st4(acc + KH + h0 + 4, p_n + 4);
      tmem_st4(acc + KH + h0 + 8, p_hn);
      tmem_st4(acc + KH + h0 + 12, p_hn + 4);
      tmem_wait_st();
      tc_fence_before();
      warp_arrive(&bars.ops_ready[a]);
      if (!mbar_wait(&bars.ph2_full[a], (i >> 1) & 1, status, 626, abort, 64)) break;
      tc_fence_after();
      uint32_t vx[16], vd[16];
      tmem_ld16(acc + 2 * KH + h0, vx);
      tmem_ld16(acc + 3 * KH + h0, vd);
      tmem_wait_ld();
      tc_fence_before();
      warp_arrive(&bars.acc_empty[a]);
      uint32_t px[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) px[j] = pk2(__uint_as_float(vx[2 * j]), __uint_as_float(vx[2 * j + 1]));
      store_T8(dXT, ld_x, row, h0, px);
      float4* go = reinterpret_cast<float4*>(gout + (size_t)row * KH + h0);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        go[q] = make_float4(dhd[4 * q] + __uint_as_float(vd[4 * q]),
                            dhd[4 * q + 1] + __uint_as_float(vd[4 * q + 1]),
                            dhd[4 * q + 2] + __uint_as_float(vd[4 * q + 2]),
                            dhd[4 * q + 3] + __uint_as_float(vd[4 * q + 3]));
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}


// ------------------------------------------------------------------------------------ H = 128
// At H = 128, W_ih and W_hh (192 KB of bf16) do not fit in shared memory beside the tiles, so
// these kernels stream them from L2 in pieces through a small TMA ring, and work on one 64-column
// half of the state at a time (a job = (tile, half hh)): the gate pre-activations of the half's
// columns h in [64 hh, 64 hh + 64) take 256 TMEM columns ([r|z] 128, Wi_n x 64, Wh_n h 64).
//   gate piece (m, ka): rows {r, z, n} x [64 hh, +64) of W_m (m = ih, hh), K-columns [64 ka, +64):
//                       192 rows x 128 B (three 64-row boxes), 24 KB
//   backward piece (m, gate): W_m^T rows h' in [0, 128), K-columns gate*H + [64 hh, +64):
//                       128 rows x 128 B, 16 KB
namespace wide {

constexpr int H = 128, NH = H / 64;
constexpr int kTileB = 128 * H * 2;          // 128 rows x H bf16: NH 64-column atoms of 16 KB
constexpr int kAtomB = 128 * 128;
constexpr int kPiece = 192 * 128;            // ring slot (gate pieces; backward pieces use 16 KB)
constexpr int kSlots = 3;                    // forward piece ring
constexpr int kSlotsB = 5;                   // backward piece ring
constexpr int kGin = 128 * 64 * 4;           // one half of the incoming gradient: 2 boxes of 16 KB
constexpr int kGates = 4 * 64;               // TMEM columns of one job's gate pre-activations

// The forward takes H = 128 or 256 (HW): HW / 64 jobs per tile, one 64-column slice each; the tile
// ring holds two stages at H = 128 and one at H = 256 (a 128-row tile of Y and E is 128 KB there).
template <int HW>
struct FwdCfg {
  static constexpr int NH = HW / 64;
  static constexpr int kTileB = 128 * HW * 2;
  static constexpr int NS = HW <= 128 ? 2 : 1;  // tile stages
  static constexpr int STAGE = 2 * kTileB;      // Y, E
  static constexpr int PIECES = NS * STAGE;
  static constexpr int SMEM = PIECES + kSlots * kPiece + 1024;
  static_assert(SMEM + 8192 <= 232448, "shared memory");
};

struct Smem {
  static constexpr int FWD_STAGE = 2 * kTileB;  // Y, E
  static constexpr int FWD_PIECES = 2 * FWD_STAGE;
  static constexpr int FWD = FWD_PIECES + kSlots * kPiece + 1024;
  static constexpr int BWD_STAGE = 2 * kTileB;       // Y, E (one stage)
  static constexpr int BWD_GIN = BWD_STAGE;          // the job's half of the incoming gradient
  static constexpr int BWD_PIECES = BWD_GIN + kGin;
  static constexpr int BWD = BWD_PIECES + kSlotsB * kPiece + 1024;
  static_assert(FWD + 4096 <= 232448 && BWD + 4096 <= 232448, "shared memory");
};

struct Bars {
  uint64_t t_full[2], t_empty[2], p_full[kSlotsB], p_empty[kSlotsB], g_full[2], g_empty[2];
  uint64_t gin_full, gin_empty, ops_ready, ph2_full, dx_empty, drain;
  uint32_t tmem_slot;
  int abort;
};

__device__ __forceinline__ void setup(Bars* b, float* bias, const float* b_ih, const float* b_hh,
                                      int warp, int Hb = H) {
  fill_gate_bias(bias, b_ih, b_hh, Hb);
  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&b->t_full[i], 1);
      mbar_init(&b->t_empty[i], kEpiWarps);
      mbar_init(&b->g_full[i], 1);
      mbar_init(&b->g_empty[i], kEpiWarps);
    }
    for (int i = 0; i < kSlotsB; ++i) { mbar_init(&b->p_full[i], 1); mbar_init(&b->p_empty[i], 1); }
    mbar_init(&b->gin_full, 1);
    mbar_init(&b->gin_empty, kEpiWarps);
    mbar_init(&b->ops_ready, kEpiWarps);
    mbar_init(&b->ph2_full, 1);
    mbar_init(&b->dx_empty, kEpiWarps);
    mbar_init(&b->drain, 1);
    b->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&b->tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  grid_dep_launch();
}

// Piece producer: for every job, the 2 NH gate pieces and (backward) the 6 backward pieces, in
// the order the MMA issuer uses them.  The weights are not written by the kernels this one may
// overlap under programmatic dependent launch (they change only between training steps).
template <int NS, int HW = H>
__device__ __forceinline__ void produce_pieces(Bars* b, uint8_t* ring, const CUtensorMap* tWih,
                                               const CUtensorMap* tWhh, const CUtensorMap* tWihT,
                                               const CUtensorMap* tWhhT, bool bwd, int n_tiles,
                                               int* status, volatile int* abort) {
  uint32_t pc = 0, issued[NS] = {};
  bool ok = true;
  auto next = [&](int bytes) -> uint8_t* {
    const int s = pc % NS;
    if (!mbar_wait(&b->p_empty[s], ((pc / NS) & 1) ^ 1, status, 631, abort, 64)) return nullptr;
    ++issued[s];
    mbar_expect_tx(&b->p_full[s], bytes);
    ++pc;
    return ring + s * kPiece;
  };
  constexpr int NHW = HW / 64;
  for (int t = blockIdx.x; t < n_tiles && ok && !*abort; t += gridDim.x) {
    for (int hh = 0; hh < NHW && ok; ++hh) {
      for (int q = 0; q < 2 * NHW && ok; ++q) {
        const int m = q / NHW, ka = q % NHW, s = pc % NS;
        uint8_t* dst = next(kPiece);
        if (!dst) { ok = false; break; }
        for (int g = 0; g < 3; ++g)
          tma_load_2d(dst + g * 64 * 128, m ? tWhh : tWih, &b->p_full[s], 64 * ka, g * HW + 64 * hh);
      }
      for (int q = 0; bwd && q < 6 && ok; ++q) {
        const int m = q / 3, g = q % 3, s = pc % NS;
        uint8_t* dst = next(128 * 128);
        if (!dst) { ok = false; break; }
        tma_load_2d(dst, m ? tWhhT : tWihT, &b->p_full[s], g * H + 64 * hh, 0);
      }
    }
  }
  if (*abort)
    for (int s = 0; s < NS; ++s)
      for (uint32_t k = 0; issued[s] && k < (1u << 22) && !mbar_try(&b->p_full[s], (issued[s] - 1) & 1); ++k) {
      }
}

// Gate pre-activations of job (tile in `stage`, half hh) into TMEM columns g0 .. g0 + 255,
// consuming 2 NH gate pieces.
template <int NS, int HW = H>
__device__ __forceinline__ bool gate_mmas(Bars* b, bool leader, uint32_t g0, uint32_t sY,
                                          uint32_t sE, uint8_t* ring, uint32_t& pc, int* status,
                                          volatile int* abort) {
  constexpr uint32_t id_rz = idesc_bf16_f32(128, 128), id_n = idesc_bf16_f32(128, 64);
  constexpr int NHW = HW / 64;
  for (int q = 0; q < 2 * NHW; ++q, ++pc) {
    const int m = q / NHW, ka = q % NHW, s = pc % NS;
    if (!mbar_wait(&b->p_full[s], (pc / NS) & 1, status, 632, abort)) return false;
    tc_fence_after();
    const uint32_t a0 = (m ? sE : sY) + ka * kAtomB, p0 = smem_u32(ring + s * kPiece);
    if (leader) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const uint64_t ad = desc_sw128_kmajor(a0 + kk * 32);
        mma_ss(g0, ad, desc_sw128_kmajor(p0 + kk * 32), id_rz, (q == 0 && kk == 0) ? 0u : 1u);
        mma_ss(g0 + 128 + 64 * m, ad, desc_sw128_kmajor(p0 + 128 * 128 + kk * 32), id_n,
               (ka == 0 && kk == 0) ? 0u : 1u);
      }
      tc_commit(&b->p_empty[s]);
    }
    __syncwarp();
  }
  return true;
}

template <int HW>
__global__ void __launch_bounds__(kThreads, 1)
    k_gru_fwd(const __grid_constant__ CUtensorMap tY, const __grid_constant__ CUtensorMap tE,
              const __grid_constant__ CUtensorMap tWih, const __grid_constant__ CUtensorMap tWhh,
              const float* __restrict__ b_ih, const float* __restrict__ b_hh,
              __nv_bfloat16* __restrict__ En, __nv_bfloat16* __restrict__ EnT, int64_t ld_T,
              int n_tiles, int n_real, int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  __shared__ Bars bars;
  using FC = FwdCfg<HW>;
  __shared__ __align__(16) float bias[4 * HW];
  volatile int* abort = &bars.abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  setup(&bars, bias, b_ih, b_hh, warp, HW);
  const uint32_t tmem = bars.tmem_slot;
  uint8_t* pieces = smem + FC::PIECES;

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------------ tile producer
    grid_dep_wait();  // Y and E are the previous kernels' output
    uint32_t issued[2] = {0, 0};
    int i = 0;
    for (int t = blockIdx.x; t < n_tiles && !*abort; t += gridDim.x, ++i) {
      const int s = i % FC::NS;
      if (!mbar_wait(&bars.t_empty[s], ((i / FC::NS) & 1) ^ 1, status, 633, abort, 64)) break;
      ++issued[s];
      uint8_t* st = smem + s * FC::STAGE;
      mbar_expect_tx(&bars.t_full[s], 2 * FC::kTileB);
      for (int a = 0; a < FC::NH; ++a) {
        tma_load_2d(st + a * kAtomB, &tY, &bars.t_full[s], 64 * a, t * 128);
        tma_load_2d(st + FC::kTileB + a * kAtomB, &tE, &bars.t_full[s], 64 * a, t * 128);
      }
    }
    if (*abort)
      for (int s = 0; s < FC::NS; ++s)
        for (uint32_t k = 0; issued[s] && k < (1u << 22) && !mbar_try(&bars.t_full[s], (issued[s] - 1) & 1); ++k) {
        }
  } else if (warp == 2 && lane == 0) {
    produce_pieces<kSlots, HW>(&bars, pieces, &tWih, &tWhh, nullptr, nullptr, false, n_tiles,
                               status, abort);
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    const bool leader = elect_one_sync();
    uint32_t pc = 0, jn = 0;
    bool ok = true;
    int i = 0;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++i) {
      const int s = i % FC::NS;
      if (!mbar_wait(&bars.t_full[s], (i / FC::NS) & 1, status, 634, abort)) break;
      const uint32_t sY = smem_u32(smem + s * FC::STAGE);
      for (int hh = 0; hh < FC::NH && ok; ++hh, ++jn) {
        const int gb = jn & 1;
        if (!mbar_wait(&bars.g_empty[gb], ((jn >> 1) & 1) ^ 1, status, 635, abort)) { ok = false; break; }
        tc_fence_after();
        if (!gate_mmas<kSlots, HW>(&bars, leader, tmem + gb * kGates, sY, sY + FC::kTileB, pieces,
                                   pc, status, abort)) {
          ok = false;
          break;
        }
        if (leader) tc_commit(&bars.g_full[gb]);
        __syncwarp();
      }
    }
    if (leader) tc_commit(&bars.drain);
    __syncwarp();
    for (uint32_t k = 0; k < (1u << 24) && !mbar_try(&bars.drain, 0); ++k) {
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------------ epilogue
    grid_dep_wait();  // outputs may still be in use by the previous kernel
    const int g = (warp - 4) / 4;
    const int r = (warp & 3) * 32 + lane;
    const uint32_t lb = (uint32_t)((warp & 3) * 32) << 16;
    uint32_t jn = 0;
    int i = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++i) {
      const int s = i % FC::NS;
      const int row = t * 128 + r;
      const bool real = row < n_real;
      const uint8_t* etile = smem + s * FC::STAGE + FC::kTileB;
      for (int hh = 0; hh < FC::NH; ++hh, ++jn) {
        const int gb = jn & 1;
        if (!mbar_wait(&bars.g_full[gb], (jn >> 1) & 1, status, 636, abort, 64)) { ok = false; break; }
        tc_fence_after();
        const uint32_t acc = tmem + lb + gb * kGates;
#pragma unroll
        for (int h8 = 0; h8 < 2; ++h8) {
          const int hs = 16 * g + 8 * h8, h = 64 * hh + hs;  // column within the half; global
          uint32_t vr[8], vz[8], vn[8], vh[8];
          tmem_ld8(acc + hs, vr);
          tmem_ld8(acc + 64 + hs, vz);
          tmem_ld8(acc + 128 + hs, vn);
          tmem_ld8(acc + 192 + hs, vh);
          tmem_wait_ld();
          float e[8];
          read_sw128_row8(etile, r, h, e);
          if (h8 == 1) {
            tc_fence_before();
            warp_arrive(&bars.g_empty[gb]);
            if (hh == FC::NH - 1) warp_arrive(&bars.t_empty[s]);
          }
          uint32_t pk[4];
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            const GateBias gb = gate_bias(bias, HW, h + 4 * q);
            float o[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const int j = 4 * q + u;
              const float rr = sigm(__uint_as_float(vr[j]) + f4(gb.r, u));
              const float zz = sigm(__uint_as_float(vz[j]) + f4(gb.z, u));
              const float nn = tanh_fast(__uint_as_float(vn[j]) + f4(gb.in, u) +
                                         rr * (__uint_as_float(vh[j]) + f4(gb.hn, u)));
              o[u] = real ? (1.f - zz) * nn + zz * e[j] : 0.f;
            }
            pk[2 * q] = pk2(o[0], o[1]);
            pk[2 * q + 1] = pk2(o[2], o[3]);
          }
          *reinterpret_cast<uint4*>(En + (size_t)row * HW + h) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
          if (EnT) store_T4(EnT, ld_T, row, h, pk);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// Gate gradients of the GRU backward at H = 256 (the GEMM path's backward: dX = dgi W_ih and
// dH += dgh W_hh then run as tensor-core GEMMs).  Per job (tile, 64-column slice hh), as in the
// forward: the gate pre-activations of the slice from streamed weight pieces into TMEM; the
// epilogue recomputes the gates, reads the incoming gradient dE(t+1) of its row and columns, and
// writes the gate gradients bf16 row-major (dgi, dgh [n][3H], the GEMMs' A operands) and
// transposed (dgi^T, dgh^T [3H][ld_T], the weight-gradient operands), and the direct term
// z * dE(t+1) (fp32, overwritten).  Padding rows get zeros.
template <int HW>
__global__ void __launch_bounds__(kThreads, 1)
    k_gru_bwd_gates(const __grid_constant__ CUtensorMap tY, const __grid_constant__ CUtensorMap tE,
                    const __grid_constant__ CUtensorMap tWih,
                    const __grid_constant__ CUtensorMap tWhh, const float* __restrict__ b_ih,
                    const float* __restrict__ b_hh, const float* __restrict__ gin,
                    float* __restrict__ gout, __nv_bfloat16* __restrict__ dgi,
                    __nv_bfloat16* __restrict__ dgh, __nv_bfloat16* __restrict__ dgiT,
                    __nv_bfloat16* __restrict__ dghT, int64_t ld_T, int n_tiles, int n_real,
                    int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  __shared__ Bars bars;
  using FC = FwdCfg<HW>;
  __shared__ __align__(16) float bias[4 * HW];
  volatile int* abort = &bars.abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  setup(&bars, bias, b_ih, b_hh, warp, HW);
  const uint32_t tmem = bars.tmem_slot;
  uint8_t* pieces = smem + FC::PIECES;

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------------ tile producer
    grid_dep_wait();  // Y, E and the incoming gradient may be the previous kernels' output
    uint32_t issued[2] = {0, 0};
    int i = 0;
    for (int t = blockIdx.x; t < n_tiles && !*abort; t += gridDim.x, ++i) {
      const int s = i % FC::NS;
      if (!mbar_wait(&bars.t_empty[s], ((i / FC::NS) & 1) ^ 1, status, 641, abort, 64)) break;
      ++issued[s];
      uint8_t* st = smem + s * FC::STAGE;
      mbar_expect_tx(&bars.t_full[s], 2 * FC::kTileB);
      for (int a = 0; a < FC::NH; ++a) {
        tma_load_2d(st + a * kAtomB, &tY, &bars.t_full[s], 64 * a, t * 128);
        tma_load_2d(st + FC::kTileB + a * kAtomB, &tE, &bars.t_full[s], 64 * a, t * 128);
      }
    }
    if (*abort)
      for (int s = 0; s < FC::NS; ++s)
        for (uint32_t k = 0; issued[s] && k < (1u << 22) && !mbar_try(&bars.t_full[s], (issued[s] - 1) & 1); ++k) {
        }
  } else if (warp == 2 && lane == 0) {
    produce_pieces<kSlots, HW>(&bars, pieces, &tWih, &tWhh, nullptr, nullptr, false, n_tiles,
                               status, abort);
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    const bool leader = elect_one_sync();
    uint32_t pc = 0, jn = 0;
    bool ok = true;
    int i = 0;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++i) {
      const int s = i % FC::NS;
      if (!mbar_wait(&bars.t_full[s], (i / FC::NS) & 1, status, 642, abort)) break;
      const uint32_t sY = smem_u32(smem + s * FC::STAGE);
      for (int hh = 0; hh < FC::NH && ok; ++hh, ++jn) {
        const int gb = jn & 1;
        if (!mbar_wait(&bars.g_empty[gb], ((jn >> 1) & 1) ^ 1, status, 643, abort)) { ok = false; break; }
        tc_fence_after();
        if (!gate_mmas<kSlots, HW>(&bars, leader, tmem + gb * kGates, sY, sY + FC::kTileB, pieces,
                                   pc, status, abort)) {
          ok = false;
          break;
        }
        if (leader) tc_commit(&bars.g_full[gb]);
        __syncwarp();
      }
    }
    if (leader) tc_commit(&bars.drain);
    __syncwarp();
    for (uint32_t k = 0; k < (1u << 24) && !mbar_try(&bars.drain, 0); ++k) {
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------------ epilogue
    grid_dep_wait();  // the outputs may still be in use by the previous kernel
    const int g = (warp - 4) / 4;
    const int r = (warp & 3) * 32 + lane;
    const uint32_t lb = (uint32_t)((warp & 3) * 32) << 16;
    uint32_t jn = 0;
    int i = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++i) {
      const int s = i % FC::NS;
      const int row = t * 128 + r;
      const bool real = row < n_real;
      const uint8_t* etile = smem + s * FC::STAGE + FC::kTileB;
      for (int hh = 0; hh < FC::NH; ++hh, ++jn) {
        const int gb = jn & 1;
        if (!mbar_wait(&bars.g_full[gb], (jn >> 1) & 1, status, 644, abort, 64)) { ok = false; break; }
        tc_fence_after();
        const uint32_t acc = tmem + lb + gb * kGates;
#pragma unroll
        for (int h8 = 0; h8 < 2; ++h8) {
          const int hs = 16 * g + 8 * h8, h = 64 * hh + hs;  // column within the slice; global
          uint32_t vr[8], vz[8], vn[8], vh[8];
          tmem_ld8(acc + hs, vr);
          tmem_ld8(acc + 64 + hs, vz);
          tmem_ld8(acc + 128 + hs, vn);
          tmem_ld8(acc + 192 + hs, vh);
          tmem_wait_ld();
          float e[8];
          read_sw128_row8(etile, r, h, e);
          if (h8 == 1) {
            tc_fence_before();
            warp_arrive(&bars.g_empty[gb]);
            if (hh == FC::NH - 1) warp_arrive(&bars.t_empty[s]);
          }
          const float4* gp = reinterpret_cast<const float4*>(gin + (size_t)row * HW + h);
          const float4 g0 = gp[0], g1 = gp[1];
          const float gv[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
          uint32_t pr[4], pz[4], pn[4], ph[4];
          float dd[8];
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            const GateBias gb4 = gate_bias(bias, HW, h + 4 * q);
            float ar[4], az[4], an[4], ahn[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const int j = 4 * q + u;
              const float rr = sigm(__uint_as_float(vr[j]) + f4(gb4.r, u));
              const float zz = sigm(__uint_as_float(vz[j]) + f4(gb4.z, u));
              const float ghn = __uint_as_float(vh[j]) + f4(gb4.hn, u);
              const float nn = tanh_fast(__uint_as_float(vn[j]) + f4(gb4.in, u) + rr * ghn);
              const float gg = real ? gv[j] : 0.f;
              const float dn = gg * (1.f - zz);
              const float dz = gg * (e[j] - nn);
              const float dan = dn * (1.f - nn * nn);
              ar[u] = dan * ghn * rr * (1.f - rr);
              az[u] = dz * zz * (1.f - zz);
              an[u] = dan;
              ahn[u] = dan * rr;
              dd[j] = gg * zz;
            }
            pr[2 * q] = pk2(ar[0], ar[1]); pr[2 * q + 1] = pk2(ar[2], ar[3]);
            pz[2 * q] = pk2(az[0], az[1]); pz[2 * q + 1] = pk2(az[2], az[3]);
            pn[2 * q] = pk2(an[0], an[1]); pn[2 * q + 1] = pk2(an[2], an[3]);
            ph[2 * q] = pk2(ahn[0], ahn[1]); ph[2 * q + 1] = pk2(ahn[2], ahn[3]);
          }
          __nv_bfloat16* di = dgi + (size_t)row * 3 * HW;
          __nv_bfloat16* dh = dgh + (size_t)row * 3 * HW;
          *reinterpret_cast<uint4*>(di + h) = make_uint4(pr[0], pr[1], pr[2], pr[3]);
          *reinterpret_cast<uint4*>(di + HW + h) = make_uint4(pz[0], pz[1], pz[2], pz[3]);
          *reinterpret_cast<uint4*>(di + 2 * HW + h) = make_uint4(pn[0], pn[1], pn[2], pn[3]);
          *reinterpret_cast<uint4*>(dh + h) = make_uint4(pr[0], pr[1], pr[2], pr[3]);
          *reinterpret_cast<uint4*>(dh + HW + h) = make_uint4(pz[0], pz[1], pz[2], pz[3]);
          *reinterpret_cast<uint4*>(dh + 2 * HW + h) = make_uint4(ph[0], ph[1], ph[2], ph[3]);
          store_T4(dgiT, ld_T, row, h, pr);
          store_T4(dgiT, ld_T, row, HW + h, pz);
          store_T4(dgiT, ld_T, row, 2 * HW + h, pn);
          store_T4(dghT, ld_T, row, h, pr);
          store_T4(dghT, ld_T, row, HW + h, pz);
          store_T4(dghT, ld_T, row, 2 * HW + h, ph);
          float4* go = reinterpret_cast<float4*>(gout + (size_t)row * HW + h);
          go[0] = make_float4(dd[0], dd[1], dd[2], dd[3]);
          go[1] = make_float4(dd[4], dd[5], dd[6], dd[7]);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// Backward.  TMEM: one job's gates (columns 0..255), dX (256..383) and dH (384..511), both
// accumulated over the tile's two halves.  Per job: gate MMAs; the epilogue forms the gate
// gradients of its columns and writes them back over the columns it read as the bf16 A operand
// (window [16 g, +16) of r: dgi_r | dgi_z pairs; of z: dgi_n | dgh_n pairs; dgh_r = dgi_r,
// dgh_z = dgi_z); then dX += dgi W_ih[half rows], dH += dgh W_hh[half rows] from the backward
// pieces.  The next job's gate MMAs wait until those products have read the gradients.
__global__ void __launch_bounds__(kThreads, 1)
    k_gru_bwd(const __grid_constant__ CUtensorMap tY, const __grid_constant__ CUtensorMap tE,
              const __grid_constant__ CUtensorMap tWih, const __grid_constant__ CUtensorMap tWhh,
              const __grid_constant__ CUtensorMap tWihT, const __grid_constant__ CUtensorMap tWhhT,
              const __grid_constant__ CUtensorMap tG, const float* __restrict__ b_ih,
              const float* __restrict__ b_hh, float* __restrict__ gout,
              __nv_bfloat16* __restrict__ dXT, int64_t ld_x, __nv_bfloat16* __restrict__ dgiT,
              __nv_bfloat16* __restrict__ dhnT, int64_t ld_g, int n_tiles, int n_real,
              int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  __shared__ Bars bars;
  __shared__ __align__(16) float bias[4 * H];
  volatile int* abort = &bars.abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  setup(&bars, bias, b_ih, b_hh, warp);
  const uint32_t tmem = bars.tmem_slot;
  uint8_t* pieces = smem + Smem::BWD_PIECES;
  constexpr uint32_t kDX = kGates, kDH = kGates + H;

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------------ tile producer (one stage)
    grid_dep_wait();  // Y, E and the incoming gradient are earlier kernels' output
    uint32_t issued = 0, gissued = 0, jn = 0;
    int i = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles && ok && !*abort; t += gridDim.x, ++i) {
      if (!mbar_wait(&bars.t_empty[0], (i & 1) ^ 1, status, 641, abort, 64)) break;
      ++issued;
      mbar_expect_tx(&bars.t_full[0], Smem::BWD_STAGE);
      for (int a = 0; a < NH; ++a) {
        tma_load_2d(smem + a * kAtomB, &tY, &bars.t_full[0], 64 * a, t * 128);
        tma_load_2d(smem + kTileB + a * kAtomB, &tE, &bars.t_full[0], 64 * a, t * 128);
      }
      // the incoming gradient one job (64-column half) at a time
      for (int hh = 0; hh < NH; ++hh, ++jn) {
        if (!mbar_wait(&bars.gin_empty, (jn & 1) ^ 1, status, 649, abort, 64)) { ok = false; break; }
        ++gissued;
        mbar_expect_tx(&bars.gin_full, kGin);
        for (int a = 0; a < 2; ++a)
          tma_load_2d(smem + Smem::BWD_GIN + a * kAtomB, &tG, &bars.gin_full, 64 * hh + 32 * a,
                      t * 128);
      }
    }
    if (*abort) {
      for (uint32_t k = 0; issued && k < (1u << 22) && !mbar_try(&bars.t_full[0], (issued - 1) & 1); ++k) {
      }
      for (uint32_t k = 0; gissued && k < (1u << 22) && !mbar_try(&bars.gin_full, (gissued - 1) & 1); ++k) {
      }
    }
  } else if (warp == 2 && lane == 0) {
    produce_pieces<kSlotsB>(&bars, pieces, &tWih, &tWhh, &tWihT, &tWhhT, true, n_tiles, status,
                            abort);
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    const bool leader = elect_one_sync();
    constexpr uint32_t id_x = idesc_bf16_f32(128, H);
    uint32_t pc = 0, jn = 0;
    bool ok = true;
    int i = 0;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++i) {
      if (!mbar_wait(&bars.t_full[0], i & 1, status, 642, abort)) break;
      const uint32_t sY = smem_u32(smem);
      for (int hh = 0; hh < NH && ok; ++hh, ++jn) {
        // the previous job's products have read the gate gradients out of columns 0..255
        if (jn > 0 && !mbar_wait(&bars.ph2_full, (jn - 1) & 1, status, 643, abort)) { ok = false; break; }
        tc_fence_after();
        if (!gate_mmas<kSlotsB>(&bars, leader, tmem, sY, sY + kTileB, pieces, pc, status, abort)) {
          ok = false;
          break;
        }
        if (leader) tc_commit(&bars.g_full[0]);
        __syncwarp();
        if (!mbar_wait(&bars.ops_ready, jn & 1, status, 644, abort)) { ok = false; break; }
        // dX and dH of the previous tile have been read out before the first job overwrites them
        if (hh == 0 && i > 0 && !mbar_wait(&bars.dx_empty, (i - 1) & 1, status, 645, abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        for (int q = 0; q < 6; ++q, ++pc) {
          const int m = q / 3, gate = q % 3, s = pc % kSlotsB;
          if (!mbar_wait(&bars.p_full[s], (pc / kSlotsB) & 1, status, 646, abort)) { ok = false; break; }
          tc_fence_after();
          const uint32_t p0 = smem_u32(pieces + s * kPiece);
          if (leader) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              const uint32_t col = gate == 2 ? 64 + 16 * kk + 8 * m : 16 * kk + 8 * gate;
              mma_ts(tmem + (m ? kDH : kDX), tmem + col, desc_sw128_kmajor(p0 + kk * 32), id_x,
                     (hh == 0 && gate == 0 && kk == 0) ? 0u : 1u);
            }
            tc_commit(&bars.p_empty[s]);
          }
          __syncwarp();
        }
        if (!ok) break;
        if (leader) tc_commit(&bars.ph2_full);
        __syncwarp();
      }
    }
    if (leader) tc_commit(&bars.drain);
    __syncwarp();
    for (uint32_t k = 0; k < (1u << 24) && !mbar_try(&bars.drain, 0); ++k) {
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------------ epilogue
    grid_dep_wait();  // outputs may still be in use by the previous kernel
    const int g = (warp - 4) / 4;
    const int r = (warp & 3) * 32 + lane;
    const uint32_t lb = (uint32_t)((warp & 3) * 32) << 16;
    const uint8_t* etile = smem + kTileB;
    const uint8_t* gtile = smem + Smem::BWD_GIN;
    uint32_t jn = 0;
    int i = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++i) {
      const int row = t * 128 + r;
      const bool real = row < n_real;
      for (int hh = 0; hh < NH; ++hh, ++jn) {
        if (!mbar_wait(&bars.g_full[0], jn & 1, status, 647, abort, 64) ||
            !mbar_wait(&bars.gin_full, jn & 1, status, 650, abort, 64)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + lb;
        uint32_t p_r[8], p_z[8], p_n[8], p_hn[8];
#pragma unroll
        for (int h8 = 0; h8 < 2; ++h8) {
          const int hs = 16 * g + 8 * h8, h = 64 * hh + hs;
          float dhd[8];  // direct term z * dE(t+1), stored now and completed with dH below
          uint32_t vr[8], vz[8], vn[8], vh[8];
          tmem_ld8(acc + hs, vr);
          tmem_ld8(acc + 64 + hs, vz);
          tmem_ld8(acc + 128 + hs, vn);
          tmem_ld8(acc + 192 + hs, vh);
          tmem_wait_ld();
          float e[8];
          read_sw128_row8(etile, r, h, e);
          float4 g4[2];
          read_sw128_f32_row8(gtile, r, hs, g4);  // column hs of the job's half
          if (h8 == 1) {
            warp_arrive(&bars.gin_empty);
            if (hh == NH - 1) warp_arrive(&bars.t_empty[0]);
          }
          const int o = 4 * h8;
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            const float4 gv = g4[q];
            const float gg[4] = {gv.x, gv.y, gv.z, gv.w};
            const GateBias gb = gate_bias(bias, H, h + 4 * q);
            float dr[4], dz[4], dn[4], dhn[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const int j = 4 * q + u;
              const float rr = sigm(__uint_as_float(vr[j]) + f4(gb.r, u));
              const float zz = sigm(__uint_as_float(vz[j]) + f4(gb.z, u));
              const float ghn = __uint_as_float(vh[j]) + f4(gb.hn, u);
              const float nn = tanh_fast(__uint_as_float(vn[j]) + f4(gb.in, u) + rr * ghn);
              const float gr = real ? gg[u] : 0.f;
              const float an = gr * (1.f - zz) * (1.f - nn * nn);
              dn[u] = an;
              dhn[u] = an * rr;
              dr[u] = an * ghn * rr * (1.f - rr);
              dz[u] = gr * (e[j] - nn) * zz * (1.f - zz);
              dhd[j] = gr * zz;
            }
            p_r[o + 2 * q] = pk2(dr[0], dr[1]); p_r[o + 2 * q + 1] = pk2(dr[2], dr[3]);
            p_z[o + 2 * q] = pk2(dz[0], dz[1]); p_z[o + 2 * q + 1] = pk2(dz[2], dz[3]);
            p_n[o + 2 * q] = pk2(dn[0], dn[1]); p_n[o + 2 * q + 1] = pk2(dn[2], dn[3]);
            p_hn[o + 2 * q] = pk2(dhn[0], dhn[1]); p_hn[o + 2 * q + 1] = pk2(dhn[2], dhn[3]);
          }
          float4* go = reinterpret_cast<float4*>(gout + (size_t)row * H + h);
          go[0] = make_float4(dhd[0], dhd[1], dhd[2], dhd[3]);
          go[1] = make_float4(dhd[4], dhd[5], dhd[6], dhd[7]);
          // gate gradients transposed for the weight-gradient GEMM: dgi rows o = gate*H + h, and
        // of dgh only the n rows (its r and z rows equal dgi's)
          store_T4(dgiT, ld_g, row, h, p_r + o);
          store_T4(dgiT + (size_t)H * ld_g, ld_g, row, h, p_z + o);
          store_T4(dgiT + (size_t)2 * H * ld_g, ld_g, row, h, p_n + o);
          store_T4(dhnT, ld_g, row, h, p_hn + o);
        }
        // in-place rewrite into the columns this warpgroup read (window 16 g of r and of z)
        const uint32_t w0 = acc + 16 * g;
        tmem_st4(w0, p_r);
        tmem_st4(w0 + 4, p_r + 4);
        tmem_st4(w0 + 8, p_z);
        tmem_st4(w0 + 12, p_z + 4);
        tmem_st4(w0 + 64, p_n);
        tmem_st4(w0 + 68, p_n + 4);
        tmem_st4(w0 + 72, p_hn);
        tmem_st4(w0 + 76, p_hn + 4);
        tmem_wait_st();
        tc_fence_before();
        warp_arrive(&bars.ops_ready);
      }
      if (!ok) break;
      // dX and dH of the whole tile are complete once the last job's products are
      if (!mbar_wait(&bars.ph2_full, (jn - 1) & 1, status, 648, abort, 64)) break;
      tc_fence_after();
#pragma unroll
      for (int hh = 0; hh < NH; ++hh) {
        const int h0 = 64 * hh + 16 * g;
        uint32_t vx[16], vd[16];
        tmem_ld16(tmem + lb + kDX + h0, vx);
        tmem_ld16(tmem + lb + kDH + h0, vd);
        tmem_wait_ld();
        if (hh == NH - 1) {
          tc_fence_before();
          warp_arrive(&bars.dx_empty);
        }
        uint32_t px[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) px[j] = pk2(__uint_as_float(vx[2 * j]), __uint_as_float(vx[2 * j + 1]));
        store_T8(dXT, ld_x, row, h0, px);
        // this thread stored the direct term of these columns above
        float4* go = reinterpret_cast<float4*>(gout + (size_t)row * H + h0);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float4 d = go[q];
          go[q] = make_float4(d.x + __uint_as_float(vd[4 * q]), d.y + __uint_as_float(vd[4 * q + 1]),
                              d.z + __uint_as_float(vd[4 * q + 2]), d.w + __uint_as_float(vd[4 * q + 3]));
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

}  // namespace wide

}  // namespace

bool gru_tc_supported(int H) { return H == 32 || H == 64 || H == wide::H; }
bool gru_fwd_tc_supported(int H) { return gru_tc_supported(H) || H == 256; }

cudaError_t gru_fwd_tc(int H, int n_pad, int n_real, const __nv_bfloat16* Y,
                       const __nv_bfloat16* E, const __nv_bfloat16* W_ih,
                       const __nv_bfloat16* W_hh, const float* b_ih, const float* b_hh,
                       __nv_bfloat16* En, __nv_bfloat16* EnT, int64_t ld_T, int* status,
                       cudaStream_t st) {
  if (!gru_fwd_tc_supported(H) || n_pad % 128) return cudaErrorInvalidValue;
  const bool w = H >= 128;
  CUtensorMap tY, tE, tWi, tWh;
  if (!make_map_ld(&tY, Y, n_pad, H, H, 128) || !make_map_ld(&tE, E, n_pad, H, H, 128) ||
      !make_map_ld(&tWi, W_ih, 3 * H, H, H, w ? 64 : 3 * H) ||
      !make_map_ld(&tWh, W_hh, 3 * H, H, H, w ? 64 : 3 * H))
    return cudaErrorInvalidValue;
  auto kern = H == 256 ? wide::k_gru_fwd<256> : H == 128 ? wide::k_gru_fwd<128>
            : H == 32 ? k_gru_fwd_tc<32> : k_gru_fwd_tc<64>;
  const int smem = H == 256 ? wide::FwdCfg<256>::SMEM : H == 128 ? wide::FwdCfg<128>::SMEM
                 : H == 32 ? GruSmem<32>::FWD : GruSmem<64>::FWD;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int n_tiles = n_pad / 128;
  const int grid = std::min(n_tiles, gemm_tn_num_sms());
  e = launch_pdl(kern, dim3(grid), dim3(kThreads), smem, st, tY, tE, tWi, tWh, b_ih, b_hh, En, EnT,
                 ld_T, n_tiles, n_real, status);
  note_launch();
  return e;
}

cudaError_t gru_bwd_gates_tc(int H, int n_pad, int n_real, const __nv_bfloat16* Y,
                             const __nv_bfloat16* E, const __nv_bfloat16* W_ih,
                             const __nv_bfloat16* W_hh, const float* b_ih, const float* b_hh,
                             const float* gin, float* gout, __nv_bfloat16* dgi,
                             __nv_bfloat16* dgh, __nv_bfloat16* dgiT, __nv_bfloat16* dghT,
                             int64_t ld_T, int* status, cudaStream_t st) {
  if (H != 256 || n_pad % 128) return cudaErrorInvalidValue;
  CUtensorMap tY, tE, tWi, tWh;
  if (!make_map_ld(&tY, Y, n_pad, H, H, 128) || !make_map_ld(&tE, E, n_pad, H, H, 128) ||
      !make_map_ld(&tWi, W_ih, 3 * H, H, H, 64) || !make_map_ld(&tWh, W_hh, 3 * H, H, H, 64))
    return cudaErrorInvalidValue;
  auto kern = wide::k_gru_bwd_gates<256>;
  const int smem = wide::FwdCfg<256>::SMEM;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int n_tiles = n_pad / 128;
  const int grid = std::min(n_tiles, gemm_tn_num_sms());
  e = launch_pdl(kern, dim3(grid), dim3(kThreads), smem, st, tY, tE, tWi, tWh, b_ih, b_hh, gin, gout,
                 dgi, dgh, dgiT, dghT, ld_T, n_tiles, n_real, status);
  note_launch();
  return e;
}

cudaError_t gru_bwd_tc(int H, int n_pad, int n_real, const __nv_bfloat16* Y,
                       const __nv_bfloat16* E, const __nv_bfloat16* W_ih,
                       const __nv_bfloat16* W_hh, const __nv_bfloat16* W_ihT,
                       const __nv_bfloat16* W_hhT, const float* b_ih, const float* b_hh,
                       const float* gin, float* gout, __nv_bfloat16* dXT, int64_t ld_x,
                       __nv_bfloat16* dgiT, __nv_bfloat16* dhnT, int64_t ld_g, int* status,
                       cudaStream_t st) {
  if (!gru_tc_supported(H) || n_pad % 128) return cudaErrorInvalidValue;
  const bool w = H == wide::H;
  CUtensorMap tY, tE, tWi, tWh, tWiT, tWhT, tG;
  // H = 64: the transposed weights are loaded whole as three 64-column boxes; H = 128: pieces of
  // 128 rows x 64 columns
  if (!make_map_ld(&tY, Y, n_pad, H, H, 128) || !make_map_ld(&tE, E, n_pad, H, H, 128) ||
      !make_map_ld(&tWi, W_ih, 3 * H, H, H, w ? 64 : 3 * H) ||
      !make_map_ld(&tWh, W_hh, 3 * H, H, H, w ? 64 : 3 * H) ||
      !make_map_ld(&tWiT, W_ihT, H, 3 * H, 3 * H, H) ||
      !make_map_ld(&tWhT, W_hhT, H, 3 * H, 3 * H, H) || !make_map_f32(&tG, gin, n_pad, H, 128))
    return cudaErrorInvalidValue;
  auto kern = w ? wide::k_gru_bwd : H == 32 ? k_gru_bwd_tc<32> : k_gru_bwd_tc<64>;
  const int smem = w ? wide::Smem::BWD : H == 32 ? GruSmem<32>::BWD : GruSmem<64>::BWD;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int n_tiles = n_pad / 128;
  const int grid = std::min(n_tiles, gemm_tn_num_sms());
  e = launch_pdl(kern, dim3(grid), dim3(kThreads), smem, st, tY, tE, tWi, tWh, tWiT, tWhT, tG, b_ih,
                 b_hh, gout, dXT, ld_x, dgiT, dhnT, ld_g, n_tiles, n_real, status);
  note_launch();
  return e;
}

}  // namespace bg

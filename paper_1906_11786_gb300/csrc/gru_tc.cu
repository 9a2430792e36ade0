// GRU cell (Cho et al.; named in Section 2 and Algorithm 1) forward and backward on tcgen05, one
// 128-row tile of nodes per CTA.  Gate convention: rows r, z, n of W_ih / W_hh;
//   r = sigma(Wi_r x + b_ir + Wh_r h + b_hr),  z = sigma(Wi_z x + b_iz + Wh_z h + b_hz),
//   n = tanh(Wi_n x + b_in + r (Wh_n h + b_hn)),  h' = (1 - z) n + z h,
// with x the summed messages Y and h the state E; padding rows stay 0.
//
// Pre-activations live in TMEM: [r|z] = Y Wi_rz^T + E Wh_rz^T (2H columns, both products
// accumulate into one tile), Wi_n x (H) and Wh_n h (H).  The forward epilogue applies the gates
// and writes E(t+1) row-major and transposed (the next band product's operand).  The backward
// recomputes the same products, forms the gate gradients in registers, writes them back into the
// TMEM columns it has just read as the bf16 A operand of dX = dgi W_ih and dH = dgh W_hh (chained
// MMAs), and stores dX^T (the transposed-band operand), the running state gradient and dgi^T,
// dgh^T for the weight-gradient GEMM.
#include <cuda.h>
#include <cuda_bf16.h>

#include "gemm_tc.h"
#include "gru_tc.h"
#include "kernels.h"
#include "tc_util.cuh"

namespace bg {

using namespace tc;

namespace {

constexpr int kH = 64;  // state size handled by these kernels

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15])
      : "memory");
}

__device__ __forceinline__ uint32_t pk2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float sigm(float x) { return 1.f / (1.f + __expf(-x)); }

// 32 consecutive bf16 of row r (columns c0 .. c0+31, c0 % 32 == 0) of a 128-row K-major tile
// stored with the 128-byte swizzle (16-byte chunk j of row r sits at chunk j ^ (r % 8)).
__device__ __forceinline__ void read_sw128_row32(const uint8_t* tile, int r, int c0, float* out) {
  const uint8_t* row = tile + (c0 / 64) * 128 * 128 + r * 128;
  const int j0 = (c0 % 64) / 8;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint4 v = *reinterpret_cast<const uint4*>(row + (((j0 + q) ^ (r & 7)) << 4));
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      out[q * 8 + 2 * e] = __uint_as_float(w[e] << 16);
      out[q * 8 + 2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
    }
  }
}

struct GruSmem {
  static constexpr int TILE = 128 * 128;           // 128 rows x 64 bf16
  static constexpr int W = 3 * kH * 128;           // [3H][H] bf16
  static constexpr int WT = 3 * kH * 128;          // [H][3H] bf16 as three 64-column atoms
  static constexpr int OFF_Y = 0, OFF_E = TILE, OFF_WIH = 2 * TILE, OFF_WHH = OFF_WIH + W;
  static constexpr int OFF_WIHT = OFF_WHH + W, OFF_WHHT = OFF_WIHT + WT;
  static constexpr int FWD = OFF_WIHT + 1024 + 1024;
  static constexpr int BWD = OFF_WHHT + WT + 1024 + 1024;
};

// Issues [r|z], Wi_n x, Wh_n h for the tile (K = H = 64: four K=16 steps).
__device__ __forceinline__ void gru_gate_mmas(uint32_t tmem, uint32_t sY, uint32_t sE, uint32_t sWih,
                                              uint32_t sWhh) {
  constexpr uint32_t id_rz = idesc_bf16_f32(128, 2 * kH), id_h = idesc_bf16_f32(128, kH);
#pragma unroll
  for (int kk = 0; kk < 4; ++kk) {
    const uint64_t aY = desc_sw128_kmajor(sY + kk * 32), aE = desc_sw128_kmajor(sE + kk * 32);
    mma_ss(tmem + 0, aY, desc_sw128_kmajor(sWih + kk * 32), id_rz, kk > 0);
    mma_ss(tmem + 0, aE, desc_sw128_kmajor(sWhh + kk * 32), id_rz, 1u);
    mma_ss(tmem + 2 * kH, aY, desc_sw128_kmajor(sWih + 2 * kH * 128 + kk * 32), id_h, kk > 0);
    mma_ss(tmem + 3 * kH, aE, desc_sw128_kmajor(sWhh + 2 * kH * 128 + kk * 32), id_h, kk > 0);
  }
}

__global__ void __launch_bounds__(128, 1)
    k_gru_fwd_tc(const __grid_constant__ CUtensorMap tY, const __grid_constant__ CUtensorMap tE,
                 const __grid_constant__ CUtensorMap tWih, const __grid_constant__ CUtensorMap tWhh,
                 const float* __restrict__ b_ih, const float* __restrict__ b_hh,
                 __nv_bfloat16* __restrict__ En, __nv_bfloat16* __restrict__ EnT, int64_t ld_T,
                 int n_real, int* status) {
  using G = GruSmem;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  __shared__ uint64_t full, done;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;
  __shared__ float bias[6 * kH];
  volatile int* abort = &abort_flag;
  const int warp = threadIdx.x >> 5, r = threadIdx.x;
  for (int t = threadIdx.x; t < 3 * kH; t += blockDim.x) {
    bias[t] = b_ih[t];
    bias[3 * kH + t] = b_hh[t];
  }
  if (threadIdx.x == 0) {
    mbar_init(&full, 1);
    mbar_init(&done, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&tmem_slot, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  const int tile = blockIdx.x;
  bool ok = true;
  if (threadIdx.x == 0) {
    mbar_expect_tx(&full, 2 * G::TILE + 2 * G::W);
    tma_load_2d(smem + G::OFF_Y, &tY, &full, 0, tile * 128);
    tma_load_2d(smem + G::OFF_E, &tE, &full, 0, tile * 128);
    tma_load_2d(smem + G::OFF_WIH, &tWih, &full, 0, 0);
    tma_load_2d(smem + G::OFF_WHH, &tWhh, &full, 0, 0);
    if (mbar_wait(&full, 0, status, 601, abort)) {
      tc_fence_after();
      gru_gate_mmas(tmem, smem_u32(smem + G::OFF_Y), smem_u32(smem + G::OFF_E),
                    smem_u32(smem + G::OFF_WIH), smem_u32(smem + G::OFF_WHH));
      tc_commit(&done);
    } else {
      for (uint32_t t = 0; t < (1u << 22) && !mbar_try(&full, 0); ++t) {
      }
    }
  }
  __syncwarp();
  ok = mbar_wait(&done, 0, status, 602, abort);
  if (ok) {
    tc_fence_after();
    const int row = tile * 128 + r;
    const uint32_t lb = (uint32_t)(warp * 32) << 16;
    const bool real = row < n_real;
#pragma unroll
    for (int h0 = 0; h0 < kH; h0 += 32) {
      uint32_t vr[32], vz[32], vn[32], vh[32];
      tmem_ld32(tmem + lb + h0, vr);
      tmem_ld32(tmem + lb + kH + h0, vz);
      tmem_ld32(tmem + lb + 2 * kH + h0, vn);
      tmem_ld32(tmem + lb + 3 * kH + h0, vh);
      tmem_wait_ld();
      float e[32];
      read_sw128_row32(smem + G::OFF_E, r, h0, e);
      uint32_t pk[16];
#pragma unroll
      for (int j = 0; j < 32; j += 2) {
        float o[2];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int h = h0 + j + u;
          const float rr = sigm(__uint_as_float(vr[j + u]) + bias[h] + bias[3 * kH + h]);
          const float zz = sigm(__uint_as_float(vz[j + u]) + bias[kH + h] + bias[4 * kH + h]);
          const float nn = tanhf(__uint_as_float(vn[j + u]) + bias[2 * kH + h] +
                                 rr * (__uint_as_float(vh[j + u]) + bias[5 * kH + h]));
          o[u] = real ? (1.f - zz) * nn + zz * e[j + u] : 0.f;
        }
        pk[j / 2] = pk2(o[0], o[1]);
      }
      uint4* d = reinterpret_cast<uint4*>(En + (size_t)row * kH + h0);
#pragma unroll
      for (int q = 0; q < 4; ++q) d[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
      if (EnT) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          __nv_bfloat16* t = EnT + (size_t)(h0 + 2 * j) * ld_T + row;
          t[0] = __ushort_as_bfloat16((unsigned short)(pk[j] & 0xFFFFu));
          t[ld_T] = __ushort_as_bfloat16((unsigned short)(pk[j] >> 16));
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

// TMEM columns of the backward kernel
constexpr int kDX = 4 * kH, kDH = 5 * kH;
// A-operand column of gate-gradient K step kk (16 values of one gate) after the in-place rewrite
__device__ __forceinline__ uint32_t dg_col(int kk, bool hidden) {
  const int gate = kk / 4, hh = (kk % 4) * 16, c = hh / 32, sb = (hh % 32) / 16;
  if (gate == 0) return c * 32 + sb * 8;
  if (gate == 1) return c * 32 + 16 + sb * 8;
  return kH + c * 32 + (hidden ? 16 : 0) + sb * 8;
}

__global__ void __launch_bounds__(128, 1)
    k_gru_bwd_tc(const __grid_constant__ CUtensorMap tY, const __grid_constant__ CUtensorMap tE,
                 const __grid_constant__ CUtensorMap tWih, const __grid_constant__ CUtensorMap tWhh,
                 const __grid_constant__ CUtensorMap tWihT, const __grid_constant__ CUtensorMap tWhhT,
                 const float* __restrict__ b_ih, const float* __restrict__ b_hh,
                 const float* __restrict__ gin, float* __restrict__ gout,
                 __nv_bfloat16* __restrict__ dXT, int64_t ld_x, __nv_bfloat16* __restrict__ dgiT,
                 __nv_bfloat16* __restrict__ dghT, int64_t ld_g, int n_real, int* status) {
  using G = GruSmem;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  __shared__ uint64_t full, done1, done2;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;
  __shared__ float bias[6 * kH];
  volatile int* abort = &abort_flag;
  const int warp = threadIdx.x >> 5, r = threadIdx.x;
  for (int t = threadIdx.x; t < 3 * kH; t += blockDim.x) {
    bias[t] = b_ih[t];
    bias[3 * kH + t] = b_hh[t];
  }
  if (threadIdx.x == 0) {
    mbar_init(&full, 1);
    mbar_init(&done1, 1);
    mbar_init(&done2, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  const int tile = blockIdx.x;
  if (threadIdx.x == 0) {
    mbar_expect_tx(&full, 2 * G::TILE + 2 * G::W + 2 * G::WT);
    tma_load_2d(smem + G::OFF_Y, &tY, &full, 0, tile * 128);
    tma_load_2d(smem + G::OFF_E, &tE, &full, 0, tile * 128);
    tma_load_2d(smem + G::OFF_WIH, &tWih, &full, 0, 0);
    tma_load_2d(smem + G::OFF_WHH, &tWhh, &full, 0, 0);
    for (int a = 0; a < 3; ++a) {
      tma_load_2d(smem + G::OFF_WIHT + a * kH * 128, &tWihT, &full, a * 64, 0);
      tma_load_2d(smem + G::OFF_WHHT + a * kH * 128, &tWhhT, &full, a * 64, 0);
    }
    if (mbar_wait(&full, 0, status, 701, abort)) {
      tc_fence_after();
      gru_gate_mmas(tmem, smem_u32(smem + G::OFF_Y), smem_u32(smem + G::OFF_E),
                    smem_u32(smem + G::OFF_WIH), smem_u32(smem + G::OFF_WHH));
      tc_commit(&done1);
    } else {
      for (uint32_t t = 0; t < (1u << 22) && !mbar_try(&full, 0); ++t) {
      }
    }
  }
  __syncwarp();
  const int row = tile * 128 + r;
  const uint32_t lb = (uint32_t)(warp * 32) << 16;
  const bool real = row < n_real;
  float dhd[kH];
  bool ok = mbar_wait(&done1, 0, status, 702, abort);
  if (ok) {
    tc_fence_after();
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      const int h0 = 32 * c;
      uint32_t vr[32], vz[32], vn[32], vh[32];
      tmem_ld32(tmem + lb + h0, vr);
      tmem_ld32(tmem + lb + kH + h0, vz);
      tmem_ld32(tmem + lb + 2 * kH + h0, vn);
      tmem_ld32(tmem + lb + 3 * kH + h0, vh);
      tmem_wait_ld();
      float e[32];
      read_sw128_row32(smem + G::OFF_E, r, h0, e);
      const float4* g4 = reinterpret_cast<const float4*>(gin + (size_t)row * kH + h0);
      uint32_t p_r[16], p_z[16], p_n[16], p_hn[16];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const float4 gv = g4[q];
        const float gg[4] = {gv.x, gv.y, gv.z, gv.w};
        float dr[4], dz[4], dn[4], dhn[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int j = 4 * q + u, h = h0 + j;
          const float rr = sigm(__uint_as_float(vr[j]) + bias[h] + bias[3 * kH + h]);
          const float zz = sigm(__uint_as_float(vz[j]) + bias[kH + h] + bias[4 * kH + h]);
          const float ghn = __uint_as_float(vh[j]) + bias[5 * kH + h];
          const float nn = tanhf(__uint_as_float(vn[j]) + bias[2 * kH + h] + rr * ghn);
          const float g = real ? gg[u] : 0.f;
          const float an = g * (1.f - zz) * (1.f - nn * nn);
          dn[u] = an;
          dhn[u] = an * rr;
          dr[u] = an * ghn * rr * (1.f - rr);
          dz[u] = g * (e[j] - nn) * zz * (1.f - zz);
          dhd[h] = g * zz;
        }
        p_r[2 * q] = pk2(dr[0], dr[1]); p_r[2 * q + 1] = pk2(dr[2], dr[3]);
        p_z[2 * q] = pk2(dz[0], dz[1]); p_z[2 * q + 1] = pk2(dz[2], dz[3]);
        p_n[2 * q] = pk2(dn[0], dn[1]); p_n[2 * q + 1] = pk2(dn[2], dn[3]);
        p_hn[2 * q] = pk2(dhn[0], dhn[1]); p_hn[2 * q + 1] = pk2(dhn[2], dhn[3]);
      }
      // in-place rewrite into the columns read above (this chunk's windows only)
      tmem_st16(tmem + lb + c * 32, p_r);
      tmem_st16(tmem + lb + c * 32 + 16, p_z);
      tmem_st16(tmem + lb + kH + c * 32, p_n);
      tmem_st16(tmem + lb + kH + c * 32 + 16, p_hn);
      // gate gradients transposed for the weight-gradient GEMM: rows o = gate*H + h
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int h = h0 + 2 * j;
        const uint32_t w4[4] = {p_r[j], p_z[j], p_n[j], p_hn[j]};
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const unsigned short b_r = (unsigned short)(u ? w4[0] >> 16 : w4[0] & 0xFFFFu);
          const unsigned short b_z = (unsigned short)(u ? w4[1] >> 16 : w4[1] & 0xFFFFu);
          const unsigned short b_n = (unsigned short)(u ? w4[2] >> 16 : w4[2] & 0xFFFFu);
          const unsigned short b_hn = (unsigned short)(u ? w4[3] >> 16 : w4[3] & 0xFFFFu);
          const size_t col = (size_t)row;
          dgiT[(size_t)(h + u) * ld_g + col] = __ushort_as_bfloat16(b_r);
          dgiT[(size_t)(kH + h + u) * ld_g + col] = __ushort_as_bfloat16(b_z);
          dgiT[(size_t)(2 * kH + h + u) * ld_g + col] = __ushort_as_bfloat16(b_n);
          dghT[(size_t)(h + u) * ld_g + col] = __ushort_as_bfloat16(b_r);
          dghT[(size_t)(kH + h + u) * ld_g + col] = __ushort_as_bfloat16(b_z);
          dghT[(size_t)(2 * kH + h + u) * ld_g + col] = __ushort_as_bfloat16(b_hn);
        }
      }
    }
    tmem_wait_st();
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && ok && !*abort) {
    tc_fence_after();
    constexpr uint32_t id_h = idesc_bf16_f32(128, kH);
    const uint32_t sIT = smem_u32(smem + G::OFF_WIHT), sHT = smem_u32(smem + G::OFF_WHHT);
#pragma unroll
    for (int kk = 0; kk < 12; ++kk) {
      const uint32_t boff = (kk / 4) * kH * 128 + (kk % 4) * 32;
      mma_ts(tmem + kDX, tmem + dg_col(kk, false), desc_sw128_kmajor(sIT + boff), id_h, kk > 0);
      mma_ts(tmem + kDH, tmem + dg_col(kk, true), desc_sw128_kmajor(sHT + boff), id_h, kk > 0);
    }
    tc_commit(&done2);
  }
  __syncwarp();
  if (ok && mbar_wait(&done2, 0, status, 703, abort)) {
    tc_fence_after();
#pragma unroll
    for (int h0 = 0; h0 < kH; h0 += 32) {
      uint32_t vx[32], vd[32];
      tmem_ld32(tmem + lb + kDX + h0, vx);
      tmem_ld32(tmem + lb + kDH + h0, vd);
      tmem_wait_ld();
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const uint32_t w = pk2(__uint_as_float(vx[2 * j]), __uint_as_float(vx[2 * j + 1]));
        __nv_bfloat16* t = dXT + (size_t)(h0 + 2 * j) * ld_x + row;
        t[0] = __ushort_as_bfloat16((unsigned short)(w & 0xFFFFu));
        t[ld_x] = __ushort_as_bfloat16((unsigned short)(w >> 16));
      }
      float4* go = reinterpret_cast<float4*>(gout + (size_t)row * kH + h0);
#pragma unroll
      for (int q = 0; q < 8; ++q)
        go[q] = make_float4(dhd[h0 + 4 * q] + __uint_as_float(vd[4 * q]),
                            dhd[h0 + 4 * q + 1] + __uint_as_float(vd[4 * q + 1]),
                            dhd[h0 + 4 * q + 2] + __uint_as_float(vd[4 * q + 2]),
                            dhd[h0 + 4 * q + 3] + __uint_as_float(vd[4 * q + 3]));
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

}  // namespace

bool gru_tc_supported(int H) { return H == kH; }

cudaError_t gru_fwd_tc(int n_pad, int n_real, const __nv_bfloat16* Y, const __nv_bfloat16* E,
                       const __nv_bfloat16* W_ih, const __nv_bfloat16* W_hh, const float* b_ih,
                       const float* b_hh, __nv_bfloat16* En, __nv_bfloat16* EnT, int64_t ld_T,
                       int* status, cudaStream_t st) {
  CUtensorMap tY, tE, tWi, tWh;
  if (!make_map_ld(&tY, Y, n_pad, kH, kH, 128) || !make_map_ld(&tE, E, n_pad, kH, kH, 128) ||
      !make_map_ld(&tWi, W_ih, 3 * kH, kH, kH, 3 * kH) ||
      !make_map_ld(&tWh, W_hh, 3 * kH, kH, kH, 3 * kH))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(k_gru_fwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       GruSmem::FWD);
  if (e != cudaSuccess) return e;
  k_gru_fwd_tc<<<n_pad / 128, 128, GruSmem::FWD, st>>>(tY, tE, tWi, tWh, b_ih, b_hh, En, EnT, ld_T,
                                                      n_real, status);
  note_launch();
  return cudaGetLastError();
}

cudaError_t gru_bwd_tc(int n_pad, int n_real, const __nv_bfloat16* Y, const __nv_bfloat16* E,
                       const __nv_bfloat16* W_ih, const __nv_bfloat16* W_hh,
                       const __nv_bfloat16* W_ihT, const __nv_bfloat16* W_hhT, const float* b_ih,
                       const float* b_hh, const float* gin, float* gout, __nv_bfloat16* dXT,
                       int64_t ld_x, __nv_bfloat16* dgiT, __nv_bfloat16* dghT, int64_t ld_g,
                       int* status, cudaStream_t st) {
  CUtensorMap tY, tE, tWi, tWh, tWiT, tWhT;
  if (!make_map_ld(&tY, Y, n_pad, kH, kH, 128) || !make_map_ld(&tE, E, n_pad, kH, kH, 128) ||
      !make_map_ld(&tWi, W_ih, 3 * kH, kH, kH, 3 * kH) ||
      !make_map_ld(&tWh, W_hh, 3 * kH, kH, kH, 3 * kH) ||
      !make_map_ld(&tWiT, W_ihT, kH, 3 * kH, 3 * kH, kH) ||
      !make_map_ld(&tWhT, W_hhT, kH, 3 * kH, 3 * kH, kH))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(k_gru_bwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       GruSmem::BWD);
  if (e != cudaSuccess) return e;
  k_gru_bwd_tc<<<n_pad / 128, 128, GruSmem::BWD, st>>>(tY, tE, tWi, tWh, tWiT, tWhT, b_ih, b_hh,
                                                      gin, gout, dXT, ld_x, dgiT, dghT, ld_g,
                                                      n_real, status);
  note_launch();
  return cudaGetLastError();
}

}  // namespace bg

// Tensor-core (tcgen05 / TMEM / TMA) band contractions for sm_103a.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"

namespace bg {

// True when the fused tensor-core kernels handle (dtype, H, S, P) for this plan.
bool band_tc_supported(const bg_plan* p, int dtype, int H);
size_t band_tc_fwd_ws_bytes(const bg_plan* p, int dtype, int H);
size_t band_tc_bwd_ws_bytes(const bg_plan* p, int dtype, int H);
// Y = sum_p A_p (E W_p + b_p), bf16 operands, fp32 accumulation and output.
cudaError_t band_tc_fwd(const bg_plan* p, int H, const void* E, const void* W, const float* b,
                        float* Y, char* ws, size_t ws_bytes, int* status, cudaStream_t st);
// dE (+)= sum_p (A_p^T dY) W_p^T, dW_p (+)= E^T A_p^T dY, db_p (+)= colsum(A_p^T dY).
cudaError_t band_tc_bwd(const bg_plan* p, int H, const void* E, const void* W, const float* dY,
                        float* dE, float* dW, float* db, int accum, char* ws, size_t ws_bytes,
                        int* status, cudaStream_t st);
// The band kernel's second-product weights (band_tc_w_bytes): from W [P][H][H] bf16, the forward
// operand W_p^T (bwd = 0) or the backward operand W_p (bwd = 1), fp32 (kind::tf32 product).
size_t band_tc_w_bytes(const bg_plan* p, int H);
cudaError_t band_tc_prep_w(const bg_plan* p, int H, const void* W, int bwd, void* Wk,
                           cudaStream_t st);
// Kernel-level entry points used by the fused GGNN steps (operands already in kernel layout):
//   XT: [H][>= n_pad] bf16 transposed states (row stride ld_x); Wk: band_tc_prep_w(bwd = 0);
//   b2T: [H][64] bf16 bias split or NULL.  Outputs (each optional): out fp32 [n][H],
//   outb bf16 [n][H], outT bf16 [H][ld_outT].
//   split: fp32 scratch of band_tc_split_floats(p, H) floats (may be NULL: no tile splitting) for
//   the partial outputs of tiles that the launch splits over several CTAs.
//   addend (may be NULL): fp32 [rows_in][H], added to the Y rows of the plan's supernode in-edge
//   targets (row r gets addend[p->d_sin_slot[r]]) before the outputs are written.
size_t band_tc_split_floats(const bg_plan* p, int H);
//   b32: the fp32 bias [P][H] (or NULL) beside its split b2T; the S = 512 kernels at 64-column
//   slices add the bias in their epilogue from it.
cudaError_t band_tc_fwd_core(const bg_plan* p, int H, const __nv_bfloat16* XT, int64_t ld_x,
                             const void* Wk, const __nv_bfloat16* b2T, const float* b32,
                             float* out, __nv_bfloat16* outb, __nv_bfloat16* outT,
                             int64_t ld_outT, float* split, const float* addend, int* status,
                             cudaStream_t st);
//   dYT: [H][>= n_pad] bf16; Wk: band_tc_prep_w(bwd = 1); dE fp32 (+)=; dMT: [P*H][ld_mt] bf16.
cudaError_t band_tc_bwd_core(const bg_plan* p, int H, const __nv_bfloat16* dYT, int64_t ld_y,
                             const void* Wk, float* dE, int accumulate, __nv_bfloat16* dMT,
                             int64_t ld_mt, float* split, int* status, cudaStream_t st);
// out[c * ld_out + r] = bf16(in[r][c]) for `batch` consecutive R x Cc matrices (in fp32 or bf16;
// ld_out <= 0 means R; batches are R*Cc apart on both sides).
cudaError_t prep_transpose_bf16(const void* in, int in_is_f32, __nv_bfloat16* out, int R, int Cc,
                                int batch, cudaStream_t st, int64_t ld_out = 0);
// [H][64] 16-bit: columns p / 32+p hold the high part / remainder of b[p][h], as bf16, or as fp16
// for a plan whose in-degrees exceed 256 (the in-degree table is fp16 then; a finite |b| above
// 65504 is recorded in `status`).
cudaError_t prep_bias_split(const bg_plan* p, const float* b, __nv_bfloat16* b2T, int H,
                            int* status, cudaStream_t st);
// Builds and uploads the tensor-core path's plan data (no-op where unsupported); 0 on success.
int band_tc_upload(bg_plan* p, cudaStream_t st);
// Host side of band_tc_upload (band_tiles.cpp): the bit-interleaved window chunks of every
// 128-row tile, [n_pad / 128][P][C1][128][4] words for C1 128-column chunks per tile, in both
// orientations, and the per-row in-degrees [n_pad][64] as bf16; returns the largest in-degree.
int band_tc_host_tiles(const bg_plan* p, int C1, std::vector<uint32_t>& mi,
                       std::vector<uint32_t>& mti, std::vector<uint16_t>& deg);
// Loads (CUDA lazy loading) every kernel band_tc_fwd can launch for this plan's block size, at
// any H, on the current device.
cudaError_t band_tc_preload_fwd(const bg_plan* p);
// Frees device data the tensor-core path keeps with the plan.
void band_tc_release(bg_plan* p);

}  // namespace bg

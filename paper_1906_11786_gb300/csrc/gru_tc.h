// Fused GRU forward / backward on tcgen05 (gru_tc.cu); state size H in {32, 64, 128} (the
// forward also 256).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

namespace bg {

bool gru_tc_supported(int H);
// The forward kernel alone also takes H = 256 (weights streamed, one 64-column slice per job).
bool gru_fwd_tc_supported(int H);

// E(t+1) = GRU(Y, E) for all n_pad rows (rows >= n_real get 0); n_pad a multiple of 128.  Y, E, En: [n_pad][H] bf16;
// W_ih, W_hh: [3H][H] bf16; biases fp32 [3H]; EnT (may be NULL): [H][ld_T] bf16, transposed En.
cudaError_t gru_fwd_tc(int H, int n_pad, int n_real, const __nv_bfloat16* Y, const __nv_bfloat16* E,
                       const __nv_bfloat16* W_ih, const __nv_bfloat16* W_hh, const float* b_ih,
                       const float* b_hh, __nv_bfloat16* En, __nv_bfloat16* EnT, int64_t ld_T,
                       int* status, cudaStream_t st);

// Backward of gru_fwd_tc for one step.  gin: dL/dE(t+1) [n_pad][H] fp32.  Writes
//   gout [n_pad][H] fp32 = dL/dE(t) through the GRU (direct and W_hh terms; may alias gin),
//   dXT [H][ld_x] bf16 = (dL/dY)^T, dgiT [3H][ld_g] bf16 = input-side gate gradients transposed
//   (rows r, z, n), dhnT [H][ld_g] bf16 = the n rows of the hidden-side ones (the hidden-side r
//   and z rows equal dgi's).
// W_ihT, W_hhT: [H][3H] bf16 transposes of W_ih, W_hh.
cudaError_t gru_bwd_tc(int H, int n_pad, int n_real, const __nv_bfloat16* Y, const __nv_bfloat16* E,
                       const __nv_bfloat16* W_ih, const __nv_bfloat16* W_hh,
                       const __nv_bfloat16* W_ihT, const __nv_bfloat16* W_hhT, const float* b_ih,
                       const float* b_hh, const float* gin, float* gout, __nv_bfloat16* dXT,
                       int64_t ld_x, __nv_bfloat16* dgiT, __nv_bfloat16* dhnT, int64_t ld_g,
                       int* status, cudaStream_t st);

// Gate gradients of one GRU backward step at H = 256 (the GEMM path's backward then forms
// dX = dgi W_ih and adds dgh W_hh to gout with tensor-core GEMMs).  gin: dL/dE(t+1) [n_pad][H] fp32;
// writes gout [n_pad][H] fp32 = z * gin (overwritten), dgi, dgh [n_pad][3H] bf16 (rows r, z, n; the
// r and z blocks of dgh equal dgi's) and their transposes dgiT, dghT [3H][ld_T] bf16.
cudaError_t gru_bwd_gates_tc(int H, int n_pad, int n_real, const __nv_bfloat16* Y,
                             const __nv_bfloat16* E, const __nv_bfloat16* W_ih,
                             const __nv_bfloat16* W_hh, const float* b_ih, const float* b_hh,
                             const float* gin, float* gout, __nv_bfloat16* dgi,
                             __nv_bfloat16* dgh, __nv_bfloat16* dgiT, __nv_bfloat16* dghT,
                             int64_t ld_T, int* status, cudaStream_t st);

}  // namespace bg

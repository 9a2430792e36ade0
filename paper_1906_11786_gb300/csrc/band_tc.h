// Tensor-core (tcgen05 / TMEM / TMA) band contractions for sm_103a.
#pragma once

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
// Builds and uploads the tensor-core path's plan data (no-op where unsupported); 0 on success.
int band_tc_upload(bg_plan* p, cudaStream_t st);
// Frees device data the tensor-core path keeps with the plan.
void band_tc_release(bg_plan* p);

}  // namespace bg

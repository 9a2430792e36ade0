// Supernode edges (super.cu): the first rows and columns of the adjacency, beside the band.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"

namespace bg {

// Device copies of the plan's supernode edge lists (no-op without supernodes); 0 on success.
int super_upload(bg_plan* p, cudaStream_t st);
void super_release(bg_plan* p);
// Loads (CUDA lazy loading) the forward kernels on the current device.
cudaError_t super_preload_fwd();

// Forward: Y[v] += sum over supernode edges (u -> v, p) of E[u] W_p + b_p.  E [n_pad][H], W
// [P][H][H] (bf16 when bf16 != 0, else fp32), b [P][H] or NULL.  compact = 0: out is Y
// [n_pad][H] fp32 and the rows are added in place; compact = 1: out is [rows_in][H] and receives
// the sums (the band kernel's addend for the plan's slot table).
cudaError_t super_fwd(const bg_plan* p, int bf16, int H, const void* E, const void* W,
                      const float* b, float* out, int compact, cudaStream_t st);

// Scratch of super_bwd: W^T as fp32 and the per-(source, type) sums.
size_t super_bwd_ws_bytes(const bg_plan* p, int H);
// Backward: dE[u] += sum_p dM_p[u] W_p^T, dW_p += E[u]^T dM_p[u], db_p += dM_p[u] (db may be
// NULL) over the supernode edges, dM_p[u] = sum over edges (u -> v, p) of dY[v].  dY fp32
// [n_pad][H], or (dY NULL) dYT bf16 [H][ld].  weights_ready: ws already holds W^T from an
// earlier call with the same W (the GGNN steps reuse it).
cudaError_t super_bwd(const bg_plan* p, int bf16, int H, const void* E, const void* W,
                      const float* dY, const __nv_bfloat16* dYT, int64_t ld, float* dE, float* dW,
                      float* db, char* ws, cudaStream_t st, bool weights_ready = false);

}  // namespace bg

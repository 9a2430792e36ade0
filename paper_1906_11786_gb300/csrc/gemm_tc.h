// Split-K tcgen05 GEMM for weight-gradient reductions (gemm_tc.cu).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include <cstddef>
#include <cstdint>

namespace bg {

// Scratch floats gemm_tn needs for its split-K partial sums.
size_t gemm_tn_part_floats(int M, int N, int64_t K);

// Reduces over K (nodes, possibly several steps concatenated) the outer products
//   G[m][n] = sum_k A[m][k] B'[n][k]    A: [M][K] bf16 (row stride lda), B: [Hout][K] bf16
// where B' is B with a row of ones (row Hout) and 15 zero rows appended by the kernel, so column
// Hout of G is the row sum of A (a bias gradient).  Output (accumulate != 0 adds):
//   mode 0: out[m][n] = G[m][n] (n < Hout), bias[m] = G[m][Hout]
//   mode 1: m = p*Hout + o: out[p][n][o] = G[m][n], bias[m] = G[m][Hout]   (bias may be NULL)
// Hout in {32, 64, 128, 256}.  Deterministic: fixed split layout and summation order.
cudaError_t gemm_tn(const void* A, int64_t lda, const void* B, int64_t ldb, int M, int Hout,
                    int64_t K, int mode, float* out, float* bias, int accumulate, float* part,
                    size_t part_floats, int* status, cudaStream_t st);

// Up to four such problems with the same K and Hout in one launch (one wave over all their M
// tiles, one reduction); part_floats must cover gemm_tn_part_floats(sum of M, Hout + 16, K).
struct TNProblem {
  const void* A;
  int64_t lda;
  const void* B;
  int64_t ldb;
  int M;
  int mode;
  float* out;
  float* bias;
};
cudaError_t gemm_tn_multi(const TNProblem* problems, int n, int Hout, int64_t K, int accumulate,
                          float* part, size_t part_floats, int* status, cudaStream_t st);

// Batched TN GEMM on tcgen05 (fp32 accumulation):
//   C[b][m][n] (+)= sum_k A[b][m][k] B[b][n][k] (+ bias[b*sBias + n])
// A: [M][K] bf16, row stride lda, batch stride sA (0 = shared by all batches); B: [N][K] bf16, row
// stride ldb, batch stride sB (0 = shared); C fp32 row stride ldc, batch stride sC.  Strides in
// elements, multiples of 8; K > 0 (zero-padded to 64 by the tensor maps).
cudaError_t gemm_bf16_tn(const void* A, int64_t lda, int64_t sA, const void* B, int64_t ldb,
                         int64_t sB, int M, int N, int K, int batch, float* C, int64_t ldc,
                         int64_t sC, const float* bias, int64_t sBias, int accumulate, int* status,
                         cudaStream_t st);
// The same product (batch 1, no bias) rounded to bf16 and stored transposed: CT[n * ldT + m].  M
// even, N a multiple of 32, ldT even and >= M, CT 4-byte aligned.
cudaError_t gemm_bf16_tn_outT(const void* A, int64_t lda, const void* B, int64_t ldb, int M, int N,
                              int K, __nv_bfloat16* CT, int64_t ldT, int* status, cudaStream_t st);

// 2-D bf16 tensor map over row-major [rows][cols] with row stride ld elements; box {64, box_rows};
// 128-byte swizzle; reads outside the array return zero.
// Row-major fp32 [rows][cols] with the 128-byte swizzle, boxes of 32 columns x box_rows.
bool make_map_f32(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols,
                  uint32_t box_rows);
bool make_map_ld(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint64_t ld,
                 uint32_t box_rows);
int gemm_tn_num_sms();
// 3-D variant: [batch][rows][cols] with row stride ld and batch stride sbatch (elements).
bool make_map_3d(CUtensorMap* m, const void* base, uint64_t batch, uint64_t rows, uint64_t cols,
                 uint64_t ld, uint64_t sbatch, uint32_t box_rows);

// One block whose bounded mbarrier wait is never satisfied: it gives up after the poll cap and
// records a timeout (site 901) in `status`, the path every stalled pipeline role takes.
cudaError_t wait_selftest(int* status, cudaStream_t st);

}  // namespace bg

// Launchers of the library's CUDA kernels (device code lives in kernels_simt.cu and band_tc.cu).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

namespace bg {

// Counts every kernel this library launches (bg_launch_count).
void note_launch();

// CUDA events around a span of launches on `st`, accumulated under kernel id `kid` (BG_KID_*)
// while profiling is on (bg_profile_enable); no events otherwise.
class ProfSpan {
 public:
  ProfSpan(int kid, cudaStream_t st);
  ~ProfSpan();
  ProfSpan(const ProfSpan&) = delete;
  ProfSpan& operator=(const ProfSpan&) = delete;

 private:
  int kid_;
  cudaStream_t st_;
  cudaEvent_t a_ = nullptr, b_ = nullptr;
};

// Launches `kernel` with programmatic stream serialization: it may begin before the previous
// kernel in `st` completes and must call grid_dep_wait() before touching that kernel's data.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Generic fp32-accumulate GEMM with arbitrary element strides (covers transposed operands):
//   C[b][m][n] (+)= sum_k A(b,m,k) B(b,k,n) + bias[b*sBias + n]
// A(b,m,k) = A[b*sAb + m*sAm + k*sAk], B(b,k,n) = B[b*sBb + k*sBk + n*sBn]; C is row-major with
// leading dimension ldc and batch stride sCb.  A and B are fp32 or bf16 (a_bf16 / b_bf16).
struct Gemm {
  int M = 0, N = 0, K = 0, batch = 1;
  const void* A = nullptr;
  int a_bf16 = 0;
  int64_t sAb = 0, sAm = 0, sAk = 0;
  const void* B = nullptr;
  int b_bf16 = 0;
  int64_t sBb = 0, sBk = 0, sBn = 0;
  float* C = nullptr;
  int64_t sCb = 0, ldc = 0;
  const float* bias = nullptr;
  int64_t sBias = 0;
  int accumulate = 0;
};
// `part` (part_floats) is scratch for split-K partial sums (deterministic two-stage reduce).
cudaError_t gemm(const Gemm& g, float* part, size_t part_floats, cudaStream_t st);

cudaError_t pack_states(int bf16, const void* Eo, void* Eb, const int32_t* gather, int n_real,
                        int n_pad, int H, cudaStream_t st);
cudaError_t unpack_states(int bf16, const void* Eb, void* Eo, const int32_t* gather, int n_real,
                          int H, cudaStream_t st);

// Band aggregation over bit tiles: out[i] = sum_{slot, p, set bits c} X_p[(k+slot-1)S + c]
//   forward  (rows = targets):  X = M [P][n_pad][H], out = Y [n_pad][H]
//   backward (rows = sources):  X = dY [n_pad][H] shared by all p, out = dM [n_pad][P][H]
// Loads (CUDA lazy loading) every kernel band_fwd_gather and gemm can launch on this device.
cudaError_t preload_fwd_simt();
cudaError_t band_fwd_gather(const uint32_t* masks, const float* M, float* Y, int K, int S, int P,
                            int H, cudaStream_t st);
cudaError_t band_bwd_gather(const uint32_t* masksT, const float* dY, float* dM, int K, int S,
                            int P, int H, cudaStream_t st);

// Same as band_bwd_gather with bf16 output dM [n_pad][P][H].
cudaError_t band_bwd_gather_bf16(const uint32_t* masksT, const float* dY, __nv_bfloat16* dM, int K,
                                 int S, int P, int H, cudaStream_t st);
// Wp[h][p*H + o] = W[p][h][o] (bf16): W_p^T blocks side by side, the operand of dE = dM_cat Wp^T.
cudaError_t wperm(const void* W, __nv_bfloat16* Wp, int P, int H, cudaStream_t st);
cudaError_t f32_to_bf16(const float* x, __nv_bfloat16* y, int64_t n, cudaStream_t st);

// Wt[(p*H + o)*H + i] = W[p][i][o] (fp32)
cudaError_t transpose_weights(int bf16, const void* W, float* Wt, int P, int H, cudaStream_t st);

// column sums of X [rows][cols] (fp32) into out[cols] (+= when accumulate), deterministic
cudaError_t colsum(const float* X, int64_t rows, int cols, float* out, int accumulate, float* part,
                   size_t part_floats, cudaStream_t st);

// GRU gates (gate rows r, z, n): gi, gh [n_pad][3H] fp32 already hold W x + b and W h + b.
cudaError_t gru_fwd_gates(int bf16, const float* gi, const float* gh, const void* E, void* En,
                          int n_real, int n_pad, int H, cudaStream_t st);
// Backward gates: from dHn writes dgi, dgh [n_pad][3H] and dHd [n_pad][H] (the direct z*dHn
// term), zero on padding rows.
cudaError_t gru_bwd_gates(int bf16, const float* gi, const float* gh, const void* E,
                          const float* dHn, float* dgi, float* dgh, float* dHd, int n_real,
                          int n_pad, int H, cudaStream_t st);

// Mean-pool readout and squared loss.  pool [n_seg][H], resid [n_seg] and part
// [n_seg][kPoolSplit][H] (per-graph partial sums) are scratch; H <= 256.
constexpr int kPoolSplit = 32;
cudaError_t readout_loss(int bf16, const void* ET, const float* w_out, const float* target,
                         const int32_t* seg_off, const int32_t* seg_cnt, const int32_t* row_graph,
                         int n_seg, int n_pad, int H, float* pool, float* resid, float* part,
                         float* loss, float* dET, float* dw_out, cudaStream_t st);

cudaError_t adam(int64_t n, float* master, void* working, int working_bf16, float* m, float* v,
                 const float* grad, float lr, float b1, float b2, float eps, int step,
                 cudaStream_t st);

cudaError_t fill_zero_f32(float* p, int64_t n, cudaStream_t st);
cudaError_t add_inplace_f32(float* dst, const float* src, int64_t n, cudaStream_t st);

}  // namespace bg

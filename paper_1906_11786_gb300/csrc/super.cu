// Supernode propagation (the "supernode" primitive of Section 6): the edges with a supernode end
// -- the dense first rows and columns of the adjacency -- propagated beside the band.
//
// A supernode's row (its in-edges) and column (its out-edges) can reach every node of its graph,
// so these edges are kept out of the band tiles and propagated as edge lists grouped by node:
//   forward   Y[v] += sum_p (sum over supernode edges u -> v of type p of E[u]) W_p + cnt_p(v) b_p
//   backward  dM_p[u] = sum over supernode edges u -> v of type p of dY[v],
//             dE[u] += sum_p dM_p[u] W_p^T,  dW_p += E[u]^T dM_p[u],  db_p += dM_p[u].
// One CTA per node row with H threads (one state column each): the per-type aggregate is summed
// in a fixed edge order, then multiplied by W_p from shared memory, so every result is
// deterministic.  The weight gradients take one CTA per (type, input column), summing the
// (source, type) pairs of that type in ascending row order.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <numeric>
#include <vector>

#include "internal.h"
#include "kernels.h"
#include "super.h"

namespace bg {

namespace {

__device__ __forceinline__ float ldf(const float* p, size_t i) { return p[i]; }
__device__ __forceinline__ float ldf(const __nv_bfloat16* p, size_t i) {
  return __bfloat162float(p[i]);
}

// Forward: one CTA per target row r (position rows[r]), thread h = state column h.
template <typename TE>
__global__ void k_super_fwd(const int32_t* __restrict__ rows, const int32_t* __restrict__ off,
                            const int32_t* __restrict__ src, const int32_t* __restrict__ type,
                            const TE* __restrict__ E, const TE* __restrict__ W,
                            const float* __restrict__ b, int H, float* __restrict__ out,
                            int compact) {
  extern __shared__ float pre[];  // [H]: the current type's aggregate
  const int r = blockIdx.x, h = threadIdx.x;
  int e = off[r];
  const int e1 = off[r + 1];
  float y = 0.f;
  while (e < e1) {
    const int p = type[e];
    float acc = 0.f;
    int cnt = 0;
    for (; e < e1 && type[e] == p; ++e, ++cnt) acc += ldf(E, (size_t)src[e] * H + h);
    __syncthreads();  // the previous type's products have read pre[]
    pre[h] = acc;
    __syncthreads();
    const TE* Wp = W + (size_t)p * H * H;
    float s = 0.f;
    for (int i = 0; i < H; ++i) s += pre[i] * ldf(Wp, (size_t)i * H + h);
    y += s + (b ? (float)cnt * b[(size_t)p * H + h] : 0.f);
  }
  if (compact)
    out[(size_t)r * H + h] = y;
  else
    out[(size_t)rows[r] * H + h] += y;
}

// Backward: one CTA per source row r, thread h = state column h.  dY is fp32 [n][H] (dYT NULL)
// or bf16 transposed [H][ld] (dYT).  Wt[p][o][i] = W[p][i][o] (fp32).
__global__ void k_super_bwd(const int32_t* __restrict__ rows, const int32_t* __restrict__ poff,
                            const int32_t* __restrict__ pair_type,
                            const int32_t* __restrict__ pair_off, const int32_t* __restrict__ dst,
                            const float* __restrict__ dY, const __nv_bfloat16* __restrict__ dYT,
                            int64_t ld, const float* __restrict__ Wt, int H,
                            float* __restrict__ dE, float* __restrict__ dMs) {
  extern __shared__ float g[];  // [H]: the current pair's dM_p[u]
  const int r = blockIdx.x, h = threadIdx.x;
  float de = 0.f;
  for (int k = poff[r]; k < poff[r + 1]; ++k) {
    float acc = 0.f;
    for (int e = pair_off[k]; e < pair_off[k + 1]; ++e) {
      const int v = dst[e];
      acc += dYT ? __bfloat162float(dYT[(size_t)h * ld + v]) : dY[(size_t)v * H + h];
    }
    dMs[(size_t)k * H + h] = acc;
    __syncthreads();
    g[h] = acc;
    __syncthreads();
    const float* Wp = Wt + (size_t)pair_type[k] * H * H;
    float s = 0.f;
    for (int o = 0; o < H; ++o) s += g[o] * Wp[(size_t)o * H + h];
    de += s;
  }
  dE[(size_t)rows[r] * H + h] += de;
}

// dW_p[i][o] += sum over type-p pairs k (ascending source row) of E[row_k][i] dMs[k][o];
// db_p[o] += sum of dMs[k][o].  Grid (H, P), H threads (o).
template <typename TE>
__global__ void k_super_dw(const int32_t* __restrict__ type_off,
                           const int32_t* __restrict__ type_pairs,
                           const int32_t* __restrict__ pair_pos, const TE* __restrict__ E,
                           const float* __restrict__ dMs, int H, float* __restrict__ dW,
                           float* __restrict__ db) {
  const int i = blockIdx.x, p = blockIdx.y, o = threadIdx.x;
  float acc = 0.f, accb = 0.f;
  for (int q = type_off[p]; q < type_off[p + 1]; ++q) {
    const int k = type_pairs[q];
    const float gk = dMs[(size_t)k * H + o];
    acc += ldf(E, (size_t)pair_pos[k] * H + i) * gk;
    accb += gk;
  }
  dW[((size_t)p * H + i) * H + o] += acc;
  if (i == 0 && db) db[(size_t)p * H + o] += accb;
}

}  // namespace

int super_upload(bg_plan* p, cudaStream_t st) {
  const int64_t m = p->n_super_edges();
  if (m == 0) return 0;
  const int32_t* se = p->sup_edges.data();  // (target, source, type), sorted by target
  const int P = p->P;
  // in-edges by target row, each row's edges by (type, source)
  std::vector<int64_t> ord_in((size_t)m);
  std::iota(ord_in.begin(), ord_in.end(), 0);
  std::stable_sort(ord_in.begin(), ord_in.end(), [&](int64_t a, int64_t b) {
    if (se[3 * a] != se[3 * b]) return se[3 * a] < se[3 * b];
    if (se[3 * a + 2] != se[3 * b + 2]) return se[3 * a + 2] < se[3 * b + 2];
    return se[3 * a + 1] < se[3 * b + 1];
  });
  std::vector<int32_t> in_rows, in_off, in_src, in_type, slot((size_t)p->n_pad(), -1);
  for (int64_t q = 0; q < m; ++q) {
    const int64_t e = ord_in[(size_t)q];
    if (in_rows.empty() || in_rows.back() != se[3 * e]) {
      slot[se[3 * e]] = (int32_t)in_rows.size();
      in_rows.push_back(se[3 * e]);
      in_off.push_back((int32_t)q);
    }
    in_src.push_back(se[3 * e + 1]);
    in_type.push_back(se[3 * e + 2]);
  }
  in_off.push_back((int32_t)m);
  // out-edges by source row, each row's edges by (type, target); (row, type) pairs
  std::vector<int64_t> ord_out((size_t)m);
  std::iota(ord_out.begin(), ord_out.end(), 0);
  std::stable_sort(ord_out.begin(), ord_out.end(), [&](int64_t a, int64_t b) {
    if (se[3 * a + 1] != se[3 * b + 1]) return se[3 * a + 1] < se[3 * b + 1];
    if (se[3 * a + 2] != se[3 * b + 2]) return se[3 * a + 2] < se[3 * b + 2];
    return se[3 * a] < se[3 * b];
  });
  std::vector<int32_t> out_rows, out_poff, pair_type, pair_off, pair_pos, out_dst;
  for (int64_t q = 0; q < m; ++q) {
    const int64_t e = ord_out[(size_t)q];
    const int32_t u = se[3 * e + 1], t = se[3 * e + 2];
    const bool new_row = out_rows.empty() || out_rows.back() != u;
    if (new_row) {
      out_rows.push_back(u);
      out_poff.push_back((int32_t)pair_type.size());
    }
    if (new_row || pair_type.back() != t) {
      pair_type.push_back(t);
      pair_off.push_back((int32_t)q);
      pair_pos.push_back(u);
    }
    out_dst.push_back(se[3 * e]);
  }
  out_poff.push_back((int32_t)pair_type.size());
  pair_off.push_back((int32_t)m);
  const int32_t npairs = (int32_t)pair_type.size();
  // pairs grouped by type (stable: ascending row within a type)
  std::vector<int32_t> type_off((size_t)P + 1, 0), type_pairs((size_t)npairs);
  for (int32_t k = 0; k < npairs; ++k) ++type_off[pair_type[k] + 1];
  for (int t = 0; t < P; ++t) type_off[t + 1] += type_off[t];
  {
    std::vector<int32_t> fill(type_off.begin(), type_off.end() - 1);
    for (int32_t k = 0; k < npairs; ++k) type_pairs[fill[pair_type[k]]++] = k;
  }
  p->sup_rows_in = (int32_t)in_rows.size();
  p->sup_rows_out = (int32_t)out_rows.size();
  p->sup_pairs = npairs;
  // one allocation: [arrays in the order of the pointers below]
  std::vector<const std::vector<int32_t>*> parts = {&in_rows,  &in_off,    &in_src,   &in_type,
                                                    &slot,     &out_rows,  &out_poff, &pair_type,
                                                    &pair_off, &pair_pos,  &out_dst,  &type_off,
                                                    &type_pairs};
  std::vector<size_t> at;
  size_t words = 0;
  for (auto* v : parts) {
    at.push_back(words);
    words += (v->size() + 63) & ~(size_t)63;  // 256-byte aligned parts
  }
  std::vector<int32_t> blob(words, 0);
  for (size_t i = 0; i < parts.size(); ++i)
    std::copy(parts[i]->begin(), parts[i]->end(), blob.begin() + at[i]);
  if (cudaMalloc(&p->d_sup, words * 4) != cudaSuccess) return -1;
  int32_t* d = p->d_sup;
  p->d_sin_rows = d + at[0];
  p->d_sin_off = d + at[1];
  p->d_sin_src = d + at[2];
  p->d_sin_type = d + at[3];
  p->d_sin_slot = d + at[4];
  p->d_sout_rows = d + at[5];
  p->d_sout_poff = d + at[6];
  p->d_pair_type = d + at[7];
  p->d_pair_off = d + at[8];
  p->d_pair_row = d + at[9];
  p->d_sout_dst = d + at[10];
  p->d_type_off = d + at[11];
  p->d_type_pairs = d + at[12];
  if (cudaMemcpyAsync(d, blob.data(), words * 4, cudaMemcpyHostToDevice, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return -1;
  return 0;
}

cudaError_t super_preload_fwd() {
  cudaFuncAttributes a;
  cudaError_t e = cudaFuncGetAttributes(&a, k_super_fwd<__nv_bfloat16>);
  if (e == cudaSuccess) e = cudaFuncGetAttributes(&a, k_super_fwd<float>);
  return e;
}

void super_release(bg_plan* p) {
  cudaFree(p->d_sup);
  p->d_sup = nullptr;
  p->d_sin_rows = p->d_sin_off = p->d_sin_src = p->d_sin_type = p->d_sin_slot = nullptr;
  p->d_sout_rows = p->d_sout_poff = p->d_pair_type = p->d_pair_off = p->d_pair_row = nullptr;
  p->d_sout_dst = p->d_type_off = p->d_type_pairs = nullptr;
  p->sup_rows_in = p->sup_rows_out = p->sup_pairs = 0;
}

size_t super_bwd_ws_bytes(const bg_plan* p, int H) {
  if (!p->n_super_edges()) return 0;
  auto al = [](size_t x) { return (x + 255) & ~(size_t)255; };
  return al(sizeof(float) * (size_t)p->P * H * H) + al(sizeof(float) * (size_t)p->sup_pairs * H);
}

cudaError_t super_fwd(const bg_plan* p, int bf16, int H, const void* E, const void* W,
                      const float* b, float* out, int compact, cudaStream_t st) {
  if (!p->sup_rows_in) return cudaSuccess;
  const size_t smem = sizeof(float) * H;
  if (bf16)
    k_super_fwd<__nv_bfloat16><<<p->sup_rows_in, H, smem, st>>>(
        p->d_sin_rows, p->d_sin_off, p->d_sin_src, p->d_sin_type,
        static_cast<const __nv_bfloat16*>(E), static_cast<const __nv_bfloat16*>(W), b, H, out,
        compact);
  else
    k_super_fwd<float><<<p->sup_rows_in, H, smem, st>>>(
        p->d_sin_rows, p->d_sin_off, p->d_sin_src, p->d_sin_type, static_cast<const float*>(E),
        static_cast<const float*>(W), b, H, out, compact);
  note_launch();
  return cudaGetLastError();
}

cudaError_t super_bwd(const bg_plan* p, int bf16, int H, const void* E, const void* W,
                      const float* dY, const __nv_bfloat16* dYT, int64_t ld, float* dE, float* dW,
                      float* db, char* ws, cudaStream_t st, bool weights_ready) {
  if (!p->sup_rows_out) return cudaSuccess;
  auto al = [](size_t x) { return (x + 255) & ~(size_t)255; };
  float* Wt = reinterpret_cast<float*>(ws);
  float* dMs = reinterpret_cast<float*>(ws + al(sizeof(float) * (size_t)p->P * H * H));
  cudaError_t e = cudaSuccess;
  if (!weights_ready) e = transpose_weights(bf16, W, Wt, p->P, H, st);
  if (e != cudaSuccess) return e;
  k_super_bwd<<<p->sup_rows_out, H, sizeof(float) * H, st>>>(
      p->d_sout_rows, p->d_sout_poff, p->d_pair_type, p->d_pair_off, p->d_sout_dst, dY, dYT, ld,
      Wt, H, dE, dMs);
  note_launch();
  if (bf16)
    k_super_dw<__nv_bfloat16><<<dim3(H, p->P), H, 0, st>>>(
        p->d_type_off, p->d_type_pairs, p->d_pair_row, static_cast<const __nv_bfloat16*>(E), dMs,
        H, dW, db);
  else
    k_super_dw<float><<<dim3(H, p->P), H, 0, st>>>(p->d_type_off, p->d_type_pairs, p->d_pair_row,
                                                   static_cast<const float*>(E), dMs, H, dW, db);
  note_launch();
  return cudaGetLastError();
}

}  // namespace bg

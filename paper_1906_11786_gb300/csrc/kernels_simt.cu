// SIMT kernels of the band-GGNN path: generic strided GEMM, band aggregation over bit tiles,
// GRU gates, layout conversion, readout and Adam.  Every kernel is bounds-checked by its index
// arithmetic; none waits on another block.
#include <atomic>

#include "kernels.h"

namespace bg {

static std::atomic<long long> g_launches{0};
void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }
long long launch_total() { return g_launches.load(); }

namespace {

__device__ __forceinline__ float ld(const float* p, int64_t i) { return p[i]; }
__device__ __forceinline__ float ld(const __nv_bfloat16* p, int64_t i) {
  return __bfloat162float(p[i]);
}
__device__ __forceinline__ void st(float* p, int64_t i, float v) { p[i] = v; }
__device__ __forceinline__ void st(__nv_bfloat16* p, int64_t i, float v) {
  p[i] = __float2bfloat16_rn(v);
}

inline int grid_for(int64_t n, int threads) {
  int64_t b = (n + threads - 1) / threads;
  if (b > (1 << 20)) b = 1 << 20;
  return (int)(b < 1 ? 1 : b);
}

// ------------------------------------------------------------------------------------ GEMM
constexpr int GT = 64;   // output tile edge
constexpr int GK = 16;   // k step

template <typename TA, typename TB>
__global__ void __launch_bounds__(256) k_gemm(Gemm g, int splits, int kchunk, float* part) {
  __shared__ float As[GK][GT + 4];
  __shared__ float Bs[GK][GT + 4];
  const TA* A = static_cast<const TA*>(g.A);
  const TB* B = static_cast<const TB*>(g.B);
  const int b = blockIdx.z / splits, s = blockIdx.z % splits;
  const int m0 = blockIdx.y * GT, n0 = blockIdx.x * GT;
  const int kbeg = s * kchunk;
  const int kend = min(g.K, kbeg + kchunk);
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
  const bool a_k_fast = (g.sAk == 1);
  const bool b_n_fast = (g.sBn == 1);
  float acc[4][4];
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
  for (int k0 = kbeg; k0 < kend; k0 += GK) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      int idx = tid + 256 * q;
      int mm, kk;
      if (a_k_fast) { kk = idx % GK; mm = idx / GK; } else { mm = idx % GT; kk = idx / GT; }
      int m = m0 + mm, k = k0 + kk;
      As[kk][mm] = (m < g.M && k < kend) ? ld(A, b * g.sAb + m * g.sAm + k * g.sAk) : 0.f;
      int nn;
      if (b_n_fast) { nn = idx % GT; kk = idx / GT; } else { kk = idx % GK; nn = idx / GK; }
      int n = n0 + nn;
      k = k0 + kk;
      Bs[kk][nn] = (n < g.N && k < kend) ? ld(B, b * g.sBb + k * g.sBk + n * g.sBn) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < GK; ++kk) {
      float a[4], bb[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) a[r] = As[kk][ty * 4 + r];
#pragma unroll
      for (int c = 0; c < 4; ++c) bb[c] = Bs[kk][tx * 4 + c];
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] += a[r] * bb[c];
    }
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    int m = m0 + ty * 4 + r;
    if (m >= g.M) continue;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      int n = n0 + tx * 4 + c;
      if (n >= g.N) continue;
      if (splits == 1) {
        int64_t o = b * g.sCb + (int64_t)m * g.ldc + n;
        float v = acc[r][c] + (g.bias ? g.bias[b * g.sBias + n] : 0.f);
        g.C[o] = g.accumulate ? g.C[o] + v : v;
      } else {
        part[(((int64_t)s * g.batch + b) * g.M + m) * g.N + n] = acc[r][c];
      }
    }
  }
}

__global__ void k_gemm_reduce(Gemm g, int splits, const float* part) {
  int64_t total = (int64_t)g.batch * g.M * g.N;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    int n = (int)(t % g.N);
    int64_t bm = t / g.N;
    int m = (int)(bm % g.M);
    int b = (int)(bm / g.M);
    float v = 0.f;
    for (int s = 0; s < splits; ++s) v += part[(int64_t)s * total + t];
    if (g.bias) v += g.bias[b * g.sBias + n];
    int64_t o = b * g.sCb + (int64_t)m * g.ldc + n;
    g.C[o] = g.accumulate ? g.C[o] + v : v;
  }
}

// ------------------------------------------------------------------------------------ layout
template <typename T>
__global__ void k_pack(const T* Eo, T* Eb, const int32_t* gather, int n_real, int64_t total,
                       int H) {
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    int64_t q = t / H;
    int h = (int)(t % H);
    Eb[t] = q < n_real ? Eo[(int64_t)gather[q] * H + h] : T(0.f);
  }
}

template <typename T>
__global__ void k_unpack(const T* Eb, T* Eo, const int32_t* gather, int64_t total, int H) {
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    int64_t q = t / H;
    int h = (int)(t % H);
    Eo[(int64_t)gather[q] * H + h] = Eb[t];
  }
}

// ------------------------------------------------------------------------------------ band
// One warp per row; lanes hold columns lane + 32 q.  The mask word is read by every lane (a
// broadcast) and its set bits are walked in order, so the summation order is fixed.
__global__ void __launch_bounds__(256) k_band_fwd_gather(const uint32_t* __restrict__ masks,
                                                         const float* __restrict__ M,
                                                         float* __restrict__ Y, int K, int S,
                                                         int P, int H) {
  const int lane = threadIdx.x & 31;
  const int64_t i = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int64_t n_pad = (int64_t)K * S;
  if (i >= n_pad) return;
  const int k = (int)(i / S), r = (int)(i % S), W32 = S / 32, HQ = H / 32;
  float acc[8];
#pragma unroll
  for (int q = 0; q < 8; ++q) acc[q] = 0.f;
  for (int e = 0; e < 3; ++e) {
    const int kb = k + e - 1;
    if (kb < 0 || kb >= K) continue;
    for (int p = 0; p < P; ++p) {
      const uint32_t* row = masks + ((((int64_t)k * 3 + e) * P + p) * S + r) * W32;
      for (int w = 0; w < W32; ++w) {
        uint32_t word = row[w];
        while (word) {
          const int c = __ffs(word) - 1;
          word &= word - 1;
          const float* m = M + ((int64_t)p * n_pad + (int64_t)kb * S + w * 32 + c) * H;
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (q < HQ) acc[q] += m[lane + 32 * q];
        }
      }
    }
  }
#pragma unroll
  for (int q = 0; q < 8; ++q)
    if (q < HQ) Y[i * H + lane + 32 * q] = acc[q];
}

template <typename TO>
__global__ void __launch_bounds__(256) k_band_bwd_gather(const uint32_t* __restrict__ masksT,
                                                         const float* __restrict__ dY,
                                                         TO* __restrict__ dM, int K, int S,
                                                         int P, int H) {
  const int lane = threadIdx.x & 31;
  const int64_t j = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int64_t n_pad = (int64_t)K * S;
  if (j >= n_pad) return;
  const int kj = (int)(j / S), c = (int)(j % S), W32 = S / 32, HQ = H / 32;
  for (int p = 0; p < P; ++p) {
    float acc[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) acc[q] = 0.f;
    for (int e = 0; e < 3; ++e) {
      const int kb = kj + e - 1;
      if (kb < 0 || kb >= K) continue;
      const uint32_t* row = masksT + ((((int64_t)kj * 3 + e) * P + p) * S + c) * W32;
      for (int w = 0; w < W32; ++w) {
        uint32_t word = row[w];
        while (word) {
          const int t = __ffs(word) - 1;
          word &= word - 1;
          const float* g = dY + ((int64_t)kb * S + w * 32 + t) * H;
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (q < HQ) acc[q] += g[lane + 32 * q];
        }
      }
    }
#pragma unroll
    for (int q = 0; q < 8; ++q)
      if (q < HQ) st(dM, (j * P + p) * H + lane + 32 * q, acc[q]);
  }
}

// Wperm[h][p*H + o] = W[p][h][o]  (the [H][P*H] B operand of dE = dM_cat W_perm^T)
__global__ void k_wperm(const __nv_bfloat16* __restrict__ W, __nv_bfloat16* __restrict__ Wp, int P,
                        int H) {
  int64_t total = (int64_t)P * H * H;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int o = (int)(t % H);
    const int64_t ph = t / H;
    const int h = (int)(ph % H), p = (int)(ph / H);
    Wp[(int64_t)h * P * H + (int64_t)p * H + o] = W[t];
  }
}

__global__ void k_f32_to_bf16(const float* __restrict__ x, __nv_bfloat16* __restrict__ y, int64_t n) {
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < n;
       t += (int64_t)gridDim.x * blockDim.x)
    y[t] = __float2bfloat16_rn(x[t]);
}

// Four elements per thread: one 16-byte load, one 8-byte store (x 16-byte and y 8-byte aligned,
// n4 = n / 4 groups; the caller converts the n % 4 tail with k_f32_to_bf16).
__global__ void k_f32_to_bf16_x4(const float4* __restrict__ x, uint2* __restrict__ y, int64_t n4) {
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < n4;
       t += (int64_t)gridDim.x * blockDim.x) {
    const float4 v = x[t];
    __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
    y[t] = make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
  }
}

template <typename T>
__global__ void k_transpose_w(const T* W, float* Wt, int P, int H) {
  int64_t total = (int64_t)P * H * H;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    int i = (int)(t % H);
    int64_t po = t / H;
    int o = (int)(po % H);
    int p = (int)(po / H);
    Wt[t] = ld(W, ((int64_t)p * H + i) * H + o);
  }
}

__global__ void k_colsum_part(const float* X, int64_t rows, int cols, int64_t chunk, float* part) {
  int col = blockIdx.x * blockDim.x + threadIdx.x;
  if (col >= cols) return;
  int64_t r0 = blockIdx.y * chunk, r1 = min(rows, r0 + chunk);
  float s = 0.f;
  for (int64_t r = r0; r < r1; ++r) s += X[r * cols + col];
  part[(int64_t)blockIdx.y * cols + col] = s;
}

__global__ void k_colsum_reduce(const float* part, int splits, int cols, float* out, int accum) {
  int col = blockIdx.x * blockDim.x + threadIdx.x;
  if (col >= cols) return;
  float s = 0.f;
  for (int i = 0; i < splits; ++i) s += part[(int64_t)i * cols + col];
  out[col] = accum ? out[col] + s : s;
}

// ------------------------------------------------------------------------------------ GRU
__device__ __forceinline__ float sigm(float x) { return 1.f / (1.f + __expf(-x)); }

template <typename T>
__global__ void k_gru_fwd(const float* gi, const float* gh, const T* E, T* En, int n_real,
                          int64_t total, int H) {
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    int64_t i = t / H;
    int h = (int)(t % H);
    if (i >= n_real) { st(En, t, 0.f); continue; }
    const float* a = gi + i * 3 * H;
    const float* c = gh + i * 3 * H;
    float r = sigm(a[h] + c[h]);
    float z = sigm(a[H + h] + c[H + h]);
    float n = tanhf(a[2 * H + h] + r * c[2 * H + h]);
    st(En, t, (1.f - z) * n + z * ld(E, t));
  }
}

template <typename T>
__global__ void k_gru_bwd(const float* gi, const float* gh, const T* E, const float* dHn,
                          float* dgi, float* dgh, float* dHd, int n_real, int64_t total, int H) {
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    int64_t i = t / H;
    int h = (int)(t % H);
    float* oi = dgi + i * 3 * H;
    float* oh = dgh + i * 3 * H;
    if (i >= n_real) {
      oi[h] = oi[H + h] = oi[2 * H + h] = 0.f;
      oh[h] = oh[H + h] = oh[2 * H + h] = 0.f;
      dHd[t] = 0.f;
      continue;
    }
    const float* a = gi + i * 3 * H;
    const float* c = gh + i * 3 * H;
    float r = sigm(a[h] + c[h]);
    float z = sigm(a[H + h] + c[H + h]);
    float n = tanhf(a[2 * H + h] + r * c[2 * H + h]);
    float g = dHn[t];
    float dn = g * (1.f - z);
    float dz = g * (ld(E, t) - n);
    float dan = dn * (1.f - n * n);
    float dar = dan * c[2 * H + h] * r * (1.f - r);
    float daz = dz * z * (1.f - z);
    oi[h] = dar; oi[H + h] = daz; oi[2 * H + h] = dan;
    oh[h] = dar; oh[H + h] = daz; oh[2 * H + h] = dan * r;
    dHd[t] = g * z;
  }
}

// ------------------------------------------------------------------------------------ readout
// Mean pool in two passes so that every graph's rows are read by many blocks at once (one block
// per graph walked each graph's rows one load after another): block (g, k) sums rows
// [off + k cnt / kPoolSplit, off + (k + 1) cnt / kPoolSplit) of graph g, 256 / H rows at a time, into
// part[g][k][H]; k_pool_finish adds the kPoolSplit partial sums in a fixed order.
template <typename T>
__global__ void k_pool_part(const T* ET, const int32_t* seg_off, const int32_t* seg_cnt, int H,
                            float* part) {
  __shared__ float red[256];
  const int g = blockIdx.x, k = blockIdx.y;
  const int R = blockDim.x / H, r = threadIdx.x / H, h = threadIdx.x - r * H;
  const int64_t off = seg_off[g], cnt = seg_cnt[g];
  const int64_t r0 = off + k * cnt / kPoolSplit, r1 = off + (k + 1) * cnt / kPoolSplit;
  float s = 0.f;
  if (r < R)
    for (int64_t i = r0 + r; i < r1; i += R) s += ld(ET, i * H + h);
  red[threadIdx.x] = s;
  __syncthreads();
  if (r == 0) {
    for (int q = 1; q < R; ++q) s += red[q * H + h];
    part[((int64_t)g * kPoolSplit + k) * H + h] = s;
  }
}

__global__ void k_pool_finish(const float* part, const float* w_out, const float* target,
                              const int32_t* seg_cnt, int H, float* pool, float* resid) {
  __shared__ float red[256];
  const int g = blockIdx.x, h = threadIdx.x;
  float s = 0.f;
  if (h < H) {
    for (int k = 0; k < kPoolSplit; ++k) s += part[((int64_t)g * kPoolSplit + k) * H + h];
    s /= (float)seg_cnt[g];
    pool[(int64_t)g * H + h] = s;
  }
  red[h] = h < H ? s * w_out[h] : 0.f;
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if (h < o) red[h] += red[h + o];
    __syncthreads();
  }
  if (h == 0) resid[g] = red[0] - target[g];
}

__global__ void k_readout_tail(const float* pool, const float* resid, int n_seg, int H,
                               float* loss, float* dw_out) {
  int h = threadIdx.x;
  if (h < H) {
    float s = 0.f;
    for (int g = 0; g < n_seg; ++g) s += resid[g] * pool[(int64_t)g * H + h];
    dw_out[h] = s;
  }
  if (h == 0) {
    float L = 0.f;
    for (int g = 0; g < n_seg; ++g) L += 0.5f * resid[g] * resid[g];
    *loss = L;
  }
}

// dE(T) of the readout, one warp per row (no per-element division of the flat index).
__global__ void k_readout_grad(const float* w_out, const float* resid, const int32_t* seg_cnt,
                               const int32_t* row_graph, int64_t n_rows, int H, float* dET) {
  const int64_t i = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
  if (i >= n_rows) return;
  const int g = row_graph[i];
  float* d = dET + i * H;
  for (int h = threadIdx.x & 31; h < H; h += 32)
    d[h] = g < 0 ? 0.f : resid[g] * w_out[h] / (float)seg_cnt[g];
}

// ------------------------------------------------------------------------------------ Adam
__global__ void k_adam(int64_t n, float* p, __nv_bfloat16* wb, float* wf, float* m, float* v,
                       const float* g, float lr, float b1, float b2, float eps, float c1, float c2) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    float gi = g[i];
    float mi = b1 * m[i] + (1.f - b1) * gi;
    float vi = b2 * v[i] + (1.f - b2) * gi * gi;
    m[i] = mi;
    v[i] = vi;
    float pi = p[i] - lr * (mi / c1) / (sqrtf(vi / c2) + eps);
    p[i] = pi;
    if (wb) wb[i] = __float2bfloat16_rn(pi);
    if (wf) wf[i] = pi;
  }
}

__global__ void k_zero(float* p, int64_t n) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    p[i] = 0.f;
}

__global__ void k_add(float* d, const float* s, int64_t n) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    d[i] += s[i];
}

}  // namespace

// ====================================================================================== hosts

cudaError_t gemm(const Gemm& g, float* part, size_t part_floats, cudaStream_t st) {
  if (g.M <= 0 || g.N <= 0 || g.batch <= 0) return cudaSuccess;
  int tiles = ((g.N + GT - 1) / GT) * ((g.M + GT - 1) / GT) * g.batch;
  int splits = 1;
  if (g.K > 512 && tiles < 304) {
    splits = (304 + tiles - 1) / tiles;
    splits = splits > 64 ? 64 : splits;
    int maxk = (g.K + 255) / 256;
    if (splits > maxk) splits = maxk;
    while (splits > 1 && (size_t)splits * g.batch * g.M * g.N > part_floats) --splits;
  }
  int kchunk = (g.K + splits - 1) / splits;
  kchunk = ((kchunk + GK - 1) / GK) * GK;
  splits = (g.K + kchunk - 1) / kchunk;
  if (splits < 1) splits = 1;
  dim3 grid((g.N + GT - 1) / GT, (g.M + GT - 1) / GT, g.batch * splits);
  if (g.a_bf16 && g.b_bf16)
    k_gemm<__nv_bfloat16, __nv_bfloat16><<<grid, 256, 0, st>>>(g, splits, kchunk, part);
  else if (g.a_bf16)
    k_gemm<__nv_bfloat16, float><<<grid, 256, 0, st>>>(g, splits, kchunk, part);
  else if (g.b_bf16)
    k_gemm<float, __nv_bfloat16><<<grid, 256, 0, st>>>(g, splits, kchunk, part);
  else
    k_gemm<float, float><<<grid, 256, 0, st>>>(g, splits, kchunk, part);
  note_launch();
  if (splits > 1) {
    int64_t total = (int64_t)g.batch * g.M * g.N;
    k_gemm_reduce<<<grid_for(total, 256), 256, 0, st>>>(g, splits, part);
    note_launch();
  }
  return cudaGetLastError();
}

cudaError_t pack_states(int bf16, const void* Eo, void* Eb, const int32_t* gather, int n_real,
                        int n_pad, int H, cudaStream_t st) {
  int64_t total = (int64_t)n_pad * H;
  if (bf16)
    k_pack<<<grid_for(total, 256), 256, 0, st>>>(static_cast<const __nv_bfloat16*>(Eo),
                                                 static_cast<__nv_bfloat16*>(Eb), gather, n_real,
                                                 total, H);
  else
    k_pack<<<grid_for(total, 256), 256, 0, st>>>(static_cast<const float*>(Eo),
                                                 static_cast<float*>(Eb), gather, n_real, total, H);
  note_launch();
  return cudaGetLastError();
}

cudaError_t unpack_states(int bf16, const void* Eb, void* Eo, const int32_t* gather, int n_real,
                          int H, cudaStream_t st) {
  int64_t total = (int64_t)n_real * H;
  if (total == 0) return cudaSuccess;
  if (bf16)
    k_unpack<<<grid_for(total, 256), 256, 0, st>>>(static_cast<const __nv_bfloat16*>(Eb),
                                                   static_cast<__nv_bfloat16*>(Eo), gather, total,
                                                   H);
  else
    k_unpack<<<grid_for(total, 256), 256, 0, st>>>(static_cast<const float*>(Eb),
                                                   static_cast<float*>(Eo), gather, total, H);
  note_launch();
  return cudaGetLastError();
}

cudaError_t preload_fwd_simt() {
  // CUDA loads kernels lazily, on first launch; this loads the ones the SIMT forward launches
  cudaFuncAttributes a;
  cudaError_t e = cudaSuccess;
  auto take = [&](cudaError_t r) { if (e == cudaSuccess) e = r; };
  take(cudaFuncGetAttributes(&a, k_gemm<__nv_bfloat16, __nv_bfloat16>));
  take(cudaFuncGetAttributes(&a, k_gemm<__nv_bfloat16, float>));
  take(cudaFuncGetAttributes(&a, k_gemm<float, __nv_bfloat16>));
  take(cudaFuncGetAttributes(&a, k_gemm<float, float>));
  take(cudaFuncGetAttributes(&a, k_gemm_reduce));
  take(cudaFuncGetAttributes(&a, k_band_fwd_gather));
  return e;
}

cudaError_t band_fwd_gather(const uint32_t* masks, const float* M, float* Y, int K, int S, int P,
                            int H, cudaStream_t st) {
  int64_t rows = (int64_t)K * S;
  k_band_fwd_gather<<<(unsigned)((rows + 7) / 8), 256, 0, st>>>(masks, M, Y, K, S, P, H);
  note_launch();
  return cudaGetLastError();
}

cudaError_t band_bwd_gather(const uint32_t* masksT, const float* dY, float* dM, int K, int S,
                            int P, int H, cudaStream_t st) {
  int64_t rows = (int64_t)K * S;
  k_band_bwd_gather<float><<<(unsigned)((rows + 7) / 8), 256, 0, st>>>(masksT, dY, dM, K, S, P, H);
  note_launch();
  return cudaGetLastError();
}

cudaError_t band_bwd_gather_bf16(const uint32_t* masksT, const float* dY, __nv_bfloat16* dM, int K,
                                 int S, int P, int H, cudaStream_t st) {
  int64_t rows = (int64_t)K * S;
  k_band_bwd_gather<__nv_bfloat16><<<(unsigned)((rows + 7) / 8), 256, 0, st>>>(masksT, dY, dM, K,
                                                                               S, P, H);
  note_launch();
  return cudaGetLastError();
}

cudaError_t wperm(const void* W, __nv_bfloat16* Wp, int P, int H, cudaStream_t st) {
  int64_t total = (int64_t)P * H * H;
  k_wperm<<<grid_for(total, 256), 256, 0, st>>>(static_cast<const __nv_bfloat16*>(W), Wp, P, H);
  note_launch();
  return cudaGetLastError();
}

cudaError_t f32_to_bf16(const float* x, __nv_bfloat16* y, int64_t n, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  const int64_t n4 = (reinterpret_cast<uintptr_t>(x) % 16 == 0 && reinterpret_cast<uintptr_t>(y) % 8 == 0)
                         ? n / 4 : 0;
  if (n4 > 0) {
    k_f32_to_bf16_x4<<<grid_for(n4, 256), 256, 0, st>>>(reinterpret_cast<const float4*>(x),
                                                        reinterpret_cast<uint2*>(y), n4);
    note_launch();
  }
  if (n > 4 * n4) {
    k_f32_to_bf16<<<grid_for(n - 4 * n4, 256), 256, 0, st>>>(x + 4 * n4, y + 4 * n4, n - 4 * n4);
    note_launch();
  }
  return cudaGetLastError();
}

cudaError_t transpose_weights(int bf16, const void* W, float* Wt, int P, int H, cudaStream_t st) {
  int64_t total = (int64_t)P * H * H;
  if (bf16)
    k_transpose_w<<<grid_for(total, 256), 256, 0, st>>>(static_cast<const __nv_bfloat16*>(W), Wt,
                                                        P, H);
  else
    k_transpose_w<<<grid_for(total, 256), 256, 0, st>>>(static_cast<const float*>(W), Wt, P, H);
  note_launch();
  return cudaGetLastError();
}

cudaError_t colsum(const float* X, int64_t rows, int cols, float* out, int accumulate, float* part,
                   size_t part_floats, cudaStream_t st) {
  int splits = (int)((rows + 1023) / 1024);
  if (splits > 256) splits = 256;
  while (splits > 1 && (size_t)splits * cols > part_floats) --splits;
  if (splits < 1) splits = 1;
  if ((size_t)splits * cols > part_floats) return cudaErrorInvalidValue;  // partials always used
  int64_t chunk = (rows + splits - 1) / splits;
  dim3 grid((cols + 255) / 256, splits);
  k_colsum_part<<<grid, 256, 0, st>>>(X, rows, cols, chunk, part);
  note_launch();
  k_colsum_reduce<<<(cols + 255) / 256, 256, 0, st>>>(part, splits, cols, out, accumulate);
  note_launch();
  return cudaGetLastError();
}

cudaError_t gru_fwd_gates(int bf16, const float* gi, const float* gh, const void* E, void* En,
                          int n_real, int n_pad, int H, cudaStream_t st) {
  int64_t total = (int64_t)n_pad * H;
  if (bf16)
    k_gru_fwd<<<grid_for(total, 256), 256, 0, st>>>(gi, gh, static_cast<const __nv_bfloat16*>(E),
                                                    static_cast<__nv_bfloat16*>(En), n_real,
                                                    total, H);
  else
    k_gru_fwd<<<grid_for(total, 256), 256, 0, st>>>(gi, gh, static_cast<const float*>(E),
                                                    static_cast<float*>(En), n_real, total, H);
  note_launch();
  return cudaGetLastError();
}

cudaError_t gru_bwd_gates(int bf16, const float* gi, const float* gh, const void* E,
                          const float* dHn, float* dgi, float* dgh, float* dHd, int n_real,
                          int n_pad, int H, cudaStream_t st) {
  int64_t total = (int64_t)n_pad * H;
  if (bf16)
    k_gru_bwd<<<grid_for(total, 256), 256, 0, st>>>(gi, gh, static_cast<const __nv_bfloat16*>(E),
                                                    dHn, dgi, dgh, dHd, n_real, total, H);
  else
    k_gru_bwd<<<grid_for(total, 256), 256, 0, st>>>(gi, gh, static_cast<const float*>(E), dHn, dgi,
                                                    dgh, dHd, n_real, total, H);
  note_launch();
  return cudaGetLastError();
}

cudaError_t readout_loss(int bf16, const void* ET, const float* w_out, const float* target,
                         const int32_t* seg_off, const int32_t* seg_cnt, const int32_t* row_graph,
                         int n_seg, int n_pad, int H, float* pool, float* resid, float* part,
                         float* loss, float* dET, float* dw_out, cudaStream_t st) {
  if (H < 1 || H > 256) return cudaErrorInvalidValue;
  if (n_seg > 0) {
    const dim3 grid(n_seg, kPoolSplit);
    if (bf16)
      k_pool_part<<<grid, 256, 0, st>>>(static_cast<const __nv_bfloat16*>(ET), seg_off, seg_cnt, H,
                                        part);
    else
      k_pool_part<<<grid, 256, 0, st>>>(static_cast<const float*>(ET), seg_off, seg_cnt, H, part);
    note_launch();
    k_pool_finish<<<n_seg, 256, 0, st>>>(part, w_out, target, seg_cnt, H, pool, resid);
    note_launch();
  }
  k_readout_tail<<<1, 256, 0, st>>>(pool, resid, n_seg, H, loss, dw_out);
  note_launch();
  k_readout_grad<<<(unsigned)((n_pad + 7) / 8), 256, 0, st>>>(w_out, resid, seg_cnt, row_graph,
                                                              n_pad, H, dET);
  note_launch();
  return cudaGetLastError();
}

cudaError_t adam(int64_t n, float* master, void* working, int working_bf16, float* m, float* v,
                 const float* grad, float lr, float b1, float b2, float eps, int step,
                 cudaStream_t st) {
  float c1 = 1.f - powf(b1, (float)step), c2 = 1.f - powf(b2, (float)step);
  __nv_bfloat16* wb = working_bf16 ? static_cast<__nv_bfloat16*>(working) : nullptr;
  float* wf = working_bf16 ? nullptr : static_cast<float*>(working);
  k_adam<<<grid_for(n, 256), 256, 0, st>>>(n, master, wb, wf, m, v, grad, lr, b1, b2, eps, c1, c2);
  note_launch();
  return cudaGetLastError();
}

cudaError_t fill_zero_f32(float* p, int64_t n, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  k_zero<<<grid_for(n, 256), 256, 0, st>>>(p, n);
  note_launch();
  return cudaGetLastError();
}

cudaError_t add_inplace_f32(float* dst, const float* src, int64_t n, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  k_add<<<grid_for(n, 256), 256, 0, st>>>(dst, src, n);
  note_launch();
  return cudaGetLastError();
}

}  // namespace bg

// Fused band contraction on the 5th-generation tensor cores (tcgen05, TMEM, TMA) for sm_103a.
//
// Forward (Algorithm 1's aggregate-first order, Eq. 3): for a 128-row tile of block-row k and
// every edge type p,
//     pre_p = sum_{d in -1,0,+1} A_{k,d,p} E_{k+d}        (128 x 3S  times  3S x H, fp32 in TMEM)
//     Y_k  += pre_p W_p                                     (chained MMA, A operand read from TMEM)
// and the per-type bias enters as one more product deg_k [128 x 2P] x [b_hi; b_lo] with exact
// integer in-degrees and b split into two bf16 halves (fp16 for a plan with an in-degree above
// 256, where bf16 integers stop being exact).  pre_p never leaves the SM.
// Backward (transposed band): the same kernel with the transposed tiles, dY instead of E and W_p
// instead of W_p^T gives dE_j += sum_p (A^T dY)_p W_p^T; dM_p = A_p^T dY is also written (bf16,
// transposed) for the weight gradient.
//
// The second product runs as kind::tf32 straight from the fp32 pre_p (W_p staged as fp32), so no
// thread touches pre_p between the two products and no MMA issuer waits on a conversion.  The
// band product is N = 64: at H = 128 the tile makes two passes over 64-column halves of the state,
// pass hh contracting the band with columns 64 hh .. of E and multiplying by rows 64 hh .. of W_p
// (Y = sum_p sum_hh pre_p[:, hh] W_p[hh, :]); the (half, type) jobs alternate between two
// 64-column pre_p units, so a job's band products overlap the previous job's W product.
//
// The 0/1 adjacency is the MMA's A operand.  It is stored as bits (the whole band costs
// 3 P S^2 / 8 bytes per block-row) and expanded on chip straight into tensor memory: the bits of
// each 32-column word are interleaved at upload (column 2j at bit j, column 2j+1 at bit 16+j) so
// that one AND and one multiply give the packed bf16 pair {1.0 or 0, 1.0 or 0}.
//
// Roles (128 x (2 + expander groups) threads, one CTA per SM, persistent over tiles):
//   warp 0      TMA producer: state blocks (B operand of the band product), W tiles, deg, bias
//   warp 1      TMEM allocator and band-product issuer (an elected lane of the converged warp
//               issues), one wait per job (per chunk group at S = 256)
//   warp 2      mask producer: one bulk copy per (tile, type) of the bit tiles into an SMEM ring
//   warp 3      second MMA issuer: the pre_p W_p products and the bias product, so that their
//               waits never stall the band-product stream
//   expanders   thread r of a warpgroup turns row r's mask bits into bf16 A tiles in TMEM; two
//               warpgroups taking the edge types in turn (warps 4-11)
//   converters  the last warpgroup: dM_p to global (backward), final epilogue TMEM -> global
// A tcgen05.mma of N = 64 is about as long as its issue, so any wait on the band-product
// issuer leaves the tensor pipe idle: that issuer waits once per job, on a barrier that the
// expanders (all the job's A tiles are in TMEM), the second issuer (the pre_p unit is free) and
// in the backward pass the converters complete together.
// Consumer warps signal a barrier with one arrive per warp after __syncwarp.  Waiting roles other
// than the expanders sleep between polls so that the MMA issuers keep their issue slots.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include "band_tc.h"
#include "gemm_tc.h"
#include "kernels.h"
#include "tc_util.cuh"

namespace bg {

using namespace tc;

namespace {

constexpr int kTile = 128;     // rows per tile = UMMA M
constexpr int kAtom = 64;      // bf16 per 128-byte swizzle row

// Block size S: a 128-row tile sees a window of C1 128-column chunks of the state (and of its
// bit tiles): rows [row0, row0 + 128) only couple to columns in block-rows kr - 1 .. kr + 1 of
// their own block-row kr, which all lie in [ws, ws + 128 C1) with ws = (row0 / S) S - S.
//   S <= 64: C1 = 2 (the tile spans 128 / S block-rows);  S = 128: 3;  S = 256: 6;  S = 512: 12.
__host__ __device__ constexpr int band_chunks(int S) { return S <= 64 ? 2 : 3 * (S / 128); }

template <int H, int S, bool BWD = false>
struct Cfg {
  // H > SW runs as H / SW passes over SW-column slices of the state: pass hh contracts the band
  // with columns SW hh .. SW hh + SW - 1 of E and multiplies the result by rows SW hh .. of W_p,
  // into Y.  SW = 64, or 32 at H = 32.
  static constexpr int SW = H < 64 ? 32 : 64;                 // state columns per pass
  // S = 512 at SW = 64: the 1536-node window takes 192 KB, so the kernel keeps nothing else of
  // size in shared memory: the expanders read their mask words straight from global memory (L2)
  // instead of a staged ring, W has one stage, and the bias is added in the epilogue (in-degree
  // times b in fp32) instead of by a product with staged operands
  static constexpr bool GM = S == 512 && SW == 64;
  static constexpr int NH = H / SW;
  static constexpr int C1 = band_chunks(S);                   // 128-column chunks per type
  static constexpr int ATOM_X = SW * 128;                     // 64 nodes x SW state columns
  static constexpr int XWIN = 2 * C1 * ATOM_X;                // one half's window, 64-node atoms
  static constexpr int NXB = XWIN <= 48 * 1024 ? 2 : 1;       // state-window buffers
  // W ring stages: at H <= 64, S <= 128 the small window leaves room for a deeper ring (the second
  // issuer's W stages come from L2, and it gates the release of the pre_p units); measured best
  // with four stages forward and three backward, the mask ring giving up the space
  static constexpr bool DW = H <= 64 && S <= 128;
  static constexpr int NW = GM ? 1 : (DW ? (BWD ? 3 : 4) : 2);
  // W stages hold K-columns of W_p^T as fp32 (tf32 operand) in 32-column atoms of H rows: a job's
  // 64 K-columns in one stage, or at H = 256 (64 KB) in two stages of one atom
  static constexpr int WK = H <= 128 ? SW : 32;               // K-columns per stage
  static constexpr int WJ = SW / WK;                          // stages per job
  static constexpr int WSTAGE = (WK / 32) * H * 128;
  static constexpr int DEG = kTile * 128;                     // 128 rows x 64 bf16
  static constexpr int NDEG = GM ? 0 : (NH > 1 ? 1 : 2);      // deg buffers
  static constexpr int B2 = GM ? 0 : H * 128;                 // H rows x 64 bf16
  static constexpr int OFF_X = 0;
  static constexpr int OFF_W = OFF_X + NXB * XWIN;
  static constexpr int OFF_DEG = OFF_W + NW * WSTAGE;
  static constexpr int OFF_B2 = OFF_DEG + NDEG * DEG;
  static constexpr int MSTAGE = C1 * kTile * 16;              // C1 chunks x 128 rows x 128 bits
  // mask ring stages (one job each): as many as fit beside the window, at least two
  static constexpr int NM0 = (C1 <= 3 ? (DW ? (BWD ? 6 : 4) : 8) : 4) / NH;
  static constexpr int NM = GM ? 0 : (C1 > 6 ? 2 : (NM0 > 2 ? NM0 : 2));
  // ring sizes as divisors (the GM shapes have no deg or mask ring; their code paths are off)
  static constexpr int NDEGD = NDEG > 0 ? NDEG : 1, NMD = NM > 0 ? NM : 1;
  static constexpr int OFF_M = OFF_B2 + B2;
  static constexpr int OFF_BAR = OFF_M + NM * MSTAGE;
  static constexpr int SMEM = OFF_BAR + 1024 + 1024;          // barriers + 1 KB alignment slack
  // TMEM columns: Y (H), two 64-column pre_p units used by the jobs (half, type) in turn, so that
  // a job's band products overlap the previous job's W product, then the A-tile slots
  // (a third unit for the backward at H <= 64, so that the converters' read of one job's dM_p
  // overlaps the band products of the next two, measured 2% slower at packed64: 85.7 vs 84.1 us)
  static constexpr int NB = 2;
  static constexpr int YCOL = 0;
  static constexpr int D1COL0 = H < 64 ? 64 : H;              // units start 64-column aligned
  static constexpr int ACOL = D1COL0 + NB * 64;
  static constexpr int NA = (512 - ACOL) / 64;
  // a job's chunks come in CG-chunk groups (one barrier wait each), G groups per job; a group and
  // one more A tile must fit in the NA slots (H = 256 has two slots: one chunk per group)
  static constexpr int CG = (C1 <= 3 && NA > C1) ? C1 : (NA > 3 ? 3 : NA - 1);
  static constexpr int G = C1 / CG;
  static constexpr int NT = (8 / G) * G;                      // per-group barrier ring
  static constexpr int NE = 2;                                // expander warpgroups
  static constexpr int THREADS = 128 * (2 + NE);
  static_assert(H == 32 || H == 64 || H == 128 || H == 256, "state size");
  static_assert(C1 % CG == 0 && NT % G == 0, "chunk groups");
  // the release of a job's pre_p unit is signalled on the barrier of job + NB's first group: the
  // ring must hold NB jobs' groups, or that barrier would still serve a pending job
  static_assert(NT / G >= NB, "barrier ring");
  static_assert(NA >= CG + 1 && NA <= 8, "one group of A tiles and one more must fit");
  static_assert(GM || (NM >= 2 && NM <= 8), "mask ring");
  static_assert(SMEM <= 232448, "shared memory");
};

struct Bars {
  uint64_t x_full[2], x_empty[2];
  uint64_t w_full[4], w_empty[4];
  uint64_t deg_full[2], deg_empty[2];
  uint64_t b2_full;
  // release of A slot s for the expander group that uses it next: each group waits only on its
  // own barrier, once per use, so no waiter can fall two phases behind (the groups take jobs in
  // turn, and slot uses alternate between them irregularly)
  uint64_t a_empty[8][2];
  uint64_t d1_full[4];
  uint64_t t_full[8];
  uint64_t y_full, y_empty;
  uint64_t m_full[8], m_empty[8];
  uint64_t drain, drain2;
  uint32_t tmem_base;
  int abort;
};

__device__ __forceinline__ uint32_t expand_pair(uint32_t w, int j) {
  // w holds column 2j at bit j and column 2j+1 at bit 16+j (j < 8); result packs bf16 1.0/0.0
  return (w & (0x00010001u << j)) * (0x3F80u >> j);
}

// Expands one interleaved 32-bit mask word into 16 packed bf16 pairs.
__device__ __forceinline__ void expand_word(uint32_t w, uint32_t* out) {
#pragma unroll
  for (int j = 0; j < 8; ++j) out[j] = expand_pair(w, j);
  const uint32_t w8 = w >> 8;
#pragma unroll
  for (int j = 0; j < 8; ++j) out[8 + j] = expand_pair(w8, j);
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// One arrive per warp once every lane of it is done (lanes' earlier operations are ordered
// before lane 0's arrive by the warp barrier).
__device__ __forceinline__ void warp_arrive(uint64_t* bar) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}

// Bounded wait for every MMA this thread issued (commit to an unused barrier).
__device__ __forceinline__ void drain_mmas(bool leader, uint64_t* bar) {
  if (leader) tc_commit(bar);
  __syncwarp();
  for (uint32_t t = 0; t < (1u << 24) && !mbar_try(bar, 0); ++t) {
  }
}

// Work of one launch.  Items 0 .. n_full-1 are whole tiles; when the tiles do not fill the last
// round of the grid evenly, each remaining tile is split into ksplit items over consecutive ranges
// of its jobs, which write their partial Y (fp32) to their own slice of `part`, and a fix-up
// kernel sums the slices in a fixed order into the outputs.
struct Sched {
  int n_items, n_full, ksplit, part_rows;
  float* part;  // [ksplit][part_rows][H]: partial Y of split items, rows from tile n_full on
  // forward: a row r with slot[r] >= 0 gets addend[slot[r]][:] added to its Y before the outputs
  // are written (the supernode rows' messages); NULL for none
  const float* addend;
  const int32_t* slot;
  // epilogue bias (shapes without the bias product): Y[r] += sum_p deg[r][p] b[p], the in-degrees
  // as 16-bit integers ([n][64], bf16 or, bias_f16, fp16) and b fp32 [P][H]; NULL for none
  const uint16_t* deg;
  const float* bias;
  int bias_f16;
};

// Tile and job range [j0, j1) of item w; part -1 for a whole tile, else its slice.
__device__ __forceinline__ void item_of(const Sched& sc, int w, int jobs, int& tile, int& j0,
                                        int& j1, int& part) {
  if (w < sc.n_full) {
    tile = w, j0 = 0, j1 = jobs, part = -1;
    return;
  }
  const int v = w - sc.n_full;
  tile = sc.n_full + v / sc.ksplit;
  part = v % sc.ksplit;
  j0 = part * jobs / sc.ksplit;
  j1 = (part + 1) * jobs / sc.ksplit;
}

template <int H, int S, bool BWD>
__global__ void __launch_bounds__(Cfg<H, S, BWD>::THREADS, 1)
    k_band_tc(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
              const __grid_constant__ CUtensorMap tm_deg, const __grid_constant__ CUtensorMap tm_b2,
              const uint32_t* __restrict__ maskI, float* __restrict__ out,
              __nv_bfloat16* __restrict__ outb, __nv_bfloat16* __restrict__ outT, int64_t ld_outT,
              __nv_bfloat16* __restrict__ dMT, int64_t ld_mt, const Sched sc, int P, int has_bias,
              int bias_f16, int accumulate, int* status) {
  using C = Cfg<H, S, BWD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + C::OFF_BAR);
  uint8_t* xwin = smem + C::OFF_X;
  uint8_t* wring = smem + C::OFF_W;
  uint8_t* degs = smem + C::OFF_DEG;
  uint8_t* b2s = smem + C::OFF_B2;
  uint8_t* mring = smem + C::OFF_M;
  volatile int* abort = &bars->abort;
  // A job is one (half, type) of a tile, in the order tile, half, type; job c writes pre_p unit
  // c % 2.  Chunk group gi = G c + g waits on t_full[gi % NT]: the 4 warps of the expander group
  // once its A tiles are in TMEM, and for first groups (g = 0) the release of the unit: the second
  // issuer's commit and, backward, the 4 converter warps.
  constexpr int kFree = 1 + (BWD ? 4 : 0);
  const int jobs = C::NH * P;  // per tile
  if (C::GM) has_bias = 0;     // the bias enters in the epilogue (sc.bias), not as a product
  // bias: once per tile, by the whole tile or its first slice

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->x_full[i], 1); mbar_init(&bars->x_empty[i], 1);
      mbar_init(&bars->deg_full[i], 1); mbar_init(&bars->deg_empty[i], 1);
    }
    for (int i = 0; i < 4; ++i) mbar_init(&bars->d1_full[i], 1);
    for (int i = 0; i < 4; ++i) { mbar_init(&bars->w_full[i], 1); mbar_init(&bars->w_empty[i], 1); }
    for (int i = 0; i < 8; ++i) { mbar_init(&bars->a_empty[i][0], 1); mbar_init(&bars->a_empty[i][1], 1); }
    for (int i = 0; i < 8; ++i) mbar_init(&bars->t_full[i], 4 + (i % C::G == 0 ? kFree : 0));
    mbar_init(&bars->b2_full, 1);
    mbar_init(&bars->y_full, 1);
    mbar_init(&bars->y_empty, 4);
    mbar_init(&bars->drain, 1);
    mbar_init(&bars->drain2, 1);
    for (int i = 0; i < 8; ++i) { mbar_init(&bars->m_full[i], 1); mbar_init(&bars->m_empty[i], 4); }
    bars->abort = 0;
    fence_mbar_init();
    // the first NB jobs find their pre_p unit free: stand in for the releases; likewise the first
    // use of each A slot (chunk s, job s / C1)
    for (int c = 0; c < C::NB; ++c)
      for (int a = 0; a < kFree; ++a) mbar_arrive(&bars->t_full[(c * C::G) % C::NT]);
    for (int sl = 0; sl < C::NA; ++sl) mbar_arrive(&bars->a_empty[sl][(sl / C::C1) % C::NE]);
  }
  if (warp == 1) {
    tmem_alloc(&bars->tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // TMEM is held: the next kernel in the stream may be scheduled on SMs as they free up
  grid_dep_launch();
  const uint32_t tmem = bars->tmem_base;

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------------ TMA producer
    tma_prefetch_desc(&tm_x);
    tma_prefetch_desc(&tm_w);
    if (has_bias) tma_prefetch_desc(&tm_deg);
    // the state windows, W and the bias split may be the previous kernel's output (the bit tiles
    // and in-degrees are plan data)
    grid_dep_wait();
    if (has_bias) {
      mbar_expect_tx(&bars->b2_full, C::B2);
      tma_load_2d(b2s, &tm_b2, &bars->b2_full, 0, 0);
    }
    uint32_t widx = 0, xi = 0, di = 0;
    uint32_t n_x[2] = {0, 0}, n_deg[2] = {0, 0}, n_w[4] = {0, 0, 0, 0};
    bool ok = true;
    for (int w = blockIdx.x; w < sc.n_items && ok && !*abort; w += gridDim.x) {
      int k, j0, j1, part;
      item_of(sc, w, jobs, k, j0, j1, part);
      const int row0 = k * kTile, ws = (row0 / S) * S - S;
      if (has_bias && part <= 0) {
        const int db = di % C::NDEGD;
        if (!mbar_wait(&bars->deg_empty[db], ((di / C::NDEGD) & 1) ^ 1, status, 102, abort, 64)) break;
        ++n_deg[db];
        ++di;
        mbar_expect_tx(&bars->deg_full[db], C::DEG);
        tma_load_2d(degs + db * C::DEG, &tm_deg, &bars->deg_full[db], 0, row0);
      }
      // job jb = P hh + p, stepped without dividing (the issuers' loops are on the MMA issue path)
      int hh = j0 / P, p = j0 - hh * P;
      for (int jb = j0; jb < j1 && ok; ++jb, p = p + 1 == P ? (++hh, 0) : p + 1) {
        if (jb == j0 || p == 0) {
          // the window of the job's state slice: rows ws .. ws + 128 C1 of state columns SW hh ..;
          // rows outside [0, n) arrive as zeros (TMA bounds fill)
          const int xb = xi % C::NXB;
          if (!mbar_wait(&bars->x_empty[xb], ((xi / C::NXB) & 1) ^ 1, status, 101, abort, 64)) {
            ok = false;
            break;
          }
          ++n_x[xb];
          ++xi;
          mbar_expect_tx(&bars->x_full[xb], C::XWIN);
          for (int a = 0; a < 2 * C::C1; ++a)
            tma_load_2d(xwin + xb * C::XWIN + a * C::ATOM_X, &tm_x, &bars->x_full[xb],
                        ws + a * kAtom, C::SW * hh);
        }
        // per job: K-columns SW hh .. of W_p^T in WJ stages of WK / 32 atoms
        {
          for (int wj = 0; wj < C::WJ; ++wj, ++widx) {
            const int ws2 = widx % C::NW;
            if (!mbar_wait(&bars->w_empty[ws2], ((widx / C::NW) & 1) ^ 1, status, 103, abort, 64)) {
              ok = false;
              break;
            }
            ++n_w[ws2];
            mbar_expect_tx(&bars->w_full[ws2], C::WSTAGE);
            for (int a = 0; a < C::WK / 32; ++a)
              tma_load_2d(wring + ws2 * C::WSTAGE + a * H * 128, &tm_w, &bars->w_full[ws2],
                          C::SW * hh + C::WK * wj + 32 * a, p * H);
          }
        }
      }
    }
    if (*abort) {
      // let this CTA's own copies land before shared memory is released (bounded)
      auto settle = [](uint64_t* bar, uint32_t uses) {
        if (!uses) return;
        for (uint32_t t = 0; t < (1u << 22) && !mbar_try(bar, (uses - 1) & 1); ++t) {
        }
      };
      for (int q = 0; q < 2; ++q) { settle(&bars->x_full[q], n_x[q]); settle(&bars->deg_full[q], n_deg[q]); }
      for (int q = 0; q < 4; ++q) settle(&bars->w_full[q], n_w[q]);
      if (has_bias) settle(&bars->b2_full, 1);
    }
  } else if (warp == 2 && lane == 0 && !C::GM) {
    // ------------------------------------------------------------------ mask producer
    // each job's C1 bit chunks (contiguous [C1][128][4] words of its type), NM jobs ahead of the
    // expanders; both halves of a tile read the same bits
    uint32_t midx = 0, n_m[8] = {0};
    for (int w = blockIdx.x; w < sc.n_items && !*abort; w += gridDim.x) {
      int k, j0, j1, part;
      item_of(sc, w, jobs, k, j0, j1, part);
      bool ok = true;
      int p = j0 % P;
      for (int jb = j0; jb < j1; ++jb, ++midx, p = p + 1 == P ? 0 : p + 1) {
        const int ms = midx % C::NMD;
        if (!mbar_wait(&bars->m_empty[ms], ((midx / C::NMD) & 1) ^ 1, status, 104, abort, 64)) {
          ok = false;
          break;
        }
        ++n_m[ms];
        mbar_expect_tx(&bars->m_full[ms], C::MSTAGE);
        bulk_load(mring + ms * C::MSTAGE, maskI + ((size_t)k * P + p) * C::C1 * kTile * 4,
                  C::MSTAGE, &bars->m_full[ms]);
      }
      if (!ok) break;
    }
    if (*abort)
      for (int q = 0; q < 8; ++q)
        for (uint32_t t = 0; n_m[q] && t < (1u << 22) && !mbar_try(&bars->m_full[q], (n_m[q] - 1) & 1); ++t) {
        }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ band-product issuer
    // pre_p = sum over the window chunks of A_{tile,p,j} X_j (N = SW): one t_full wait per group
    // of chunks, then an unbroken MMA stream
    const bool leader = elect_one_sync();
    constexpr uint32_t idesc = idesc_bf16_f32(kTile, C::SW);
    uint32_t c = 0, slot = 0, gi = 0, xi = 0;
    // expander group of chunk x + NA (the next user of the slot chunk x frees): job (x + NA) / C1
    // mod 2, kept as a group and a position within the job
    uint32_t nx_g = (C::NA / C::C1) & 1, nx_r = C::NA % C::C1;
    bool ok = true;
    for (int w = blockIdx.x; w < sc.n_items && ok; w += gridDim.x) {
      int k, j0, j1, part;
      item_of(sc, w, jobs, k, j0, j1, part);
      // segments of the item's jobs that share a state window (one slice each)
      for (int jb = j0; jb < j1 && ok;) {
        const int seg_end = min(j1, (jb / P + 1) * P);
        const int xb = xi % C::NXB;
        if (!mbar_wait(&bars->x_full[xb], (xi / C::NXB) & 1, status, 204, abort)) { ok = false; break; }
        ++xi;
        // descriptors differ from the window's first one only in the start-address field
        const uint64_t xdesc = desc_sw128_kmajor(smem_u32(xwin + xb * C::XWIN));
        for (; jb < seg_end && ok; ++jb, ++c) {
          const uint32_t d1 = tmem + C::D1COL0 + (c % C::NB) * 64;
          for (int g = 0; g < C::G; ++g, ++gi) {
            if (!mbar_wait(&bars->t_full[gi % C::NT], (gi / C::NT) & 1, status, 210, abort)) { ok = false; break; }
            tc_fence_after();
            for (int j = g * C::CG; j < (g + 1) * C::CG; ++j) {
              const uint32_t a = tmem + C::ACOL + slot * 64;
              const uint64_t jdesc = xdesc + (uint64_t)((2 * j * C::ATOM_X) >> 4);
              // S = 32: the tile's rows couple to window columns [0, 192) only, so the last four
              // K steps of the second chunk would multiply all-zero A tiles
              const int kk_end = (S == 32 && j == C::C1 - 1) ? 4 : kTile / 16;
#pragma unroll
              for (int kk = 0; kk < kTile / 16; ++kk)
                if (leader && kk < kk_end)
                  mma_ts(d1, a + kk * 8, jdesc + (uint64_t)(((kk / 4) * C::ATOM_X + (kk % 4) * 32) >> 4),
                         idesc, (j == 0 && kk == 0) ? 0u : 1u);
              if (leader) tc_commit(&bars->a_empty[slot][nx_g]);
              slot = slot + 1 == (uint32_t)C::NA ? 0 : slot + 1;
              if (++nx_r == (uint32_t)C::C1) { nx_r = 0; nx_g ^= 1; }
            }
          }
          if (!ok) break;
          if (leader) tc_commit(&bars->d1_full[c % C::NB]);
        }
        if (!ok) break;
        if (leader) tc_commit(&bars->x_empty[xb]);  // the segment's last job is issued
      }
    }
    drain_mmas(leader, &bars->drain);
  } else if (warp == 3) {
    // ------------------------------------------------------------------ second issuer
    // Y (+)= pre_p W_p over the jobs (kind::tf32, A = the fp32 pre_p unit in TMEM, K = the 64 rows
    // of W_p of the job's half), then the bias product
    const bool leader = elect_one_sync();
    // the bias product: in-degrees and bias halves as bf16, or as fp16 when an in-degree exceeds
    // 256 (the plan's hub rows)
    const uint32_t idesc = bias_f16 ? idesc_f16_f32(kTile, H) : idesc_bf16_f32(kTile, H);
    constexpr uint32_t idesc2 = idesc_tf32_f32(kTile, H);
    uint32_t c = 0, widx = 0, di = 0;
    bool ok = true;
    int i = 0;
    for (int w = blockIdx.x; w < sc.n_items && ok; w += gridDim.x, ++i) {
      int k, j0, j1, part;
      item_of(sc, w, jobs, k, j0, j1, part);
      for (int jb = j0; jb < j1 && ok; ++jb, ++c) {
        const int b = c % C::NB;
        if (!mbar_wait(&bars->d1_full[b], (c / C::NB) & 1, status, 208, abort) ||
            (jb == j0 && !mbar_wait(&bars->y_empty, (i & 1) ^ 1, status, 203, abort))) {
          ok = false;
          break;
        }
        for (int wj = 0; wj < C::WJ; ++wj, ++widx) {
          const int ws = widx % C::NW;
          if (!mbar_wait(&bars->w_full[ws], (widx / C::NW) & 1, status, 202, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t wbase = smem_u32(wring + ws * C::WSTAGE);
#pragma unroll
          for (int kk = 0; kk < C::WK / 8; ++kk) {
            const uint64_t bdesc = desc_sw128_kmajor(wbase + (kk / 4) * H * 128 + (kk % 4) * 32);
            if (leader) mma_ts_tf32(tmem + C::YCOL, tmem + C::D1COL0 + b * 64 + C::WK * wj + kk * 8,
                                    bdesc, idesc2, (jb == j0 && wj == 0 && kk == 0) ? 0u : 1u);
          }
          if (leader) tc_commit(&bars->w_empty[ws]);
        }
        if (!ok) break;
        // this unit is free again: part of job c + NB's first group
        if (leader) tc_commit(&bars->t_full[((c + C::NB) * C::G) % C::NT]);
      }
      if (!ok) break;
      if (has_bias && part <= 0) {
        const int db = di % C::NDEGD;
        if (!mbar_wait(&bars->deg_full[db], (di / C::NDEGD) & 1, status, 206, abort)) break;
        if (di == 0 && !mbar_wait(&bars->b2_full, 0, status, 207, abort)) break;
        ++di;
        tc_fence_after();
        const uint32_t dbase = smem_u32(degs + db * C::DEG), bbase = smem_u32(b2s);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          if (leader) mma_ss(tmem + C::YCOL, desc_sw128_kmajor(dbase + kk * 32),
                 desc_sw128_kmajor(bbase + kk * 32), idesc, 1u);
        if (leader) tc_commit(&bars->deg_empty[db]);
      }
      if (leader) tc_commit(&bars->y_full);
    }
    // a CTA whose items were all later slices of split tiles never used the bias rows it loaded:
    // let that copy land before the CTA's shared memory is released
    if (has_bias && di == 0) mbar_wait(&bars->b2_full, 0, status, 209, abort);
    drain_mmas(leader, &bars->drain2);
  } else if (warp >= 4 && warp < 4 + 4 * C::NE) {
    // ------------------------------------------------------------------ expanders
    // the two groups take the jobs in turn
    const int eg = (warp - 4) / 4;
    const int r = (threadIdx.x - 128) % 128;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    uint32_t aidx = 0, midx = 0;
    uint32_t par = 0;  // bit s: parity of this group's waits so far on A slot s
    for (int w = blockIdx.x; w < sc.n_items && !*abort; w += gridDim.x) {
      int k, j0, j1, part;
      item_of(sc, w, jobs, k, j0, j1, part);
      bool ok = true;
      for (int jb = j0; jb < j1 && ok; ++jb, ++midx) {
        if ((int)(midx % C::NE) != eg) {
          aidx += C::C1;  // the other group's job
          continue;
        }
        // one chunk: wait for its A slot, expand the row's 128 bits into bf16 pairs in TMEM, and
        // after the last chunk of a group signal the band-product issuer
        auto expand_chunk = [&](int j, const uint4 m) -> bool {
          const int slot = aidx % C::NA;
          if (!mbar_wait(&bars->a_empty[slot][eg], (par >> slot) & 1, status, 301, abort))
            return false;
          par ^= 1u << slot;
          tc_fence_after();
          uint32_t v[32];
          expand_word(m.x, v);
          expand_word(m.y, v + 16);
          tmem_st32(tmem + lane_base + C::ACOL + slot * 64, v);
          expand_word(m.z, v);
          expand_word(m.w, v + 16);
          tmem_st32(tmem + lane_base + C::ACOL + slot * 64 + 32, v);
          if ((j + 1) % C::CG == 0) {
            // all of this group's A tiles are in TMEM
            tmem_wait_st();
            tc_fence_before();
            const uint32_t gi = midx * C::G + j / C::CG;
            warp_arrive(&bars->t_full[gi % C::NT]);
          }
          ++aidx;
          return true;
        };
        // this row's mask words of the job's chunks: from the staged ring, or (GM) straight from
        // global memory in groups of four chunks, the next group requested while the current one
        // is expanded (a rolled group loop keeps the code small enough for the instruction cache)
        const int ms = C::GM ? 0 : midx % C::NMD;
        if constexpr (C::GM) {
          constexpr int QG = 4;
          static_assert(C::C1 % QG == 0, "mask prefetch groups");
          const uint4* mg = reinterpret_cast<const uint4*>(maskI) +
                            ((size_t)k * P + (jb % P)) * C::C1 * kTile + r;
          uint4 cur[QG], nxt[QG];
#pragma unroll
          for (int q = 0; q < QG; ++q) cur[q] = __ldg(mg + (size_t)q * kTile);
#pragma unroll 1
          for (int g0 = 0; g0 < C::C1 && ok; g0 += QG) {
            if (g0 + QG < C::C1) {
#pragma unroll
              for (int q = 0; q < QG; ++q) nxt[q] = __ldg(mg + (size_t)(g0 + QG + q) * kTile);
            }
#pragma unroll
            for (int q = 0; q < QG; ++q)
              if (ok && !expand_chunk(g0 + q, cur[q])) ok = false;
#pragma unroll
            for (int q = 0; q < QG; ++q) cur[q] = nxt[q];
          }
        } else {
          if (!mbar_wait(&bars->m_full[ms], (midx / C::NMD) & 1, status, 302, abort, 32)) {
            ok = false;
            break;
          }
          const uint8_t* mrow = mring + ms * C::MSTAGE + r * 16;
          for (int j = 0; j < C::C1; ++j) {
            // the words are read into registers before the slot wait, so that the shared-memory
            // load overlaps it
            const uint4 m = *reinterpret_cast<const uint4*>(mrow + j * kTile * 16);
            if (!expand_chunk(j, m)) {
              ok = false;
              break;
            }
          }
        }
        if (!ok) break;
        if (!C::GM) warp_arrive(&bars->m_empty[ms]);
      }
      if (!ok) break;
    }
  } else if (warp >= 4 + 4 * C::NE) {
    // ------------------------------------------------------------------ converters / epilogue
    grid_dep_wait();  // outputs (and the accumulated dE) may still be in use by the previous kernel
    const int r = threadIdx.x - 128 * (1 + C::NE);
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    uint32_t c = 0;
    int i = 0;
    for (int w = blockIdx.x; w < sc.n_items && !*abort; w += gridDim.x, ++i) {
      int k, j0, j1, part;
      item_of(sc, w, jobs, k, j0, j1, part);
      const int row = k * kTile + r;
      const int asl = (!BWD && sc.addend && part < 0) ? sc.slot[row] : -1;
      bool ok = true;
      int hh = j0 / P, p = j0 - hh * P;
      for (int jb = j0; BWD && jb < j1; ++jb, ++c, p = p + 1 == P ? (++hh, 0) : p + 1) {
        const int b = c % C::NB;
        if (!mbar_wait(&bars->d1_full[b], (c / C::NB) & 1, status, 401, abort, 64)) { ok = false; break; }
        tc_fence_after();
        const uint32_t col = tmem + lane_base + C::D1COL0 + b * 64;
        uint32_t v[C::SW];
        tmem_ld32(col, v);
        if constexpr (C::SW > 32) tmem_ld32(col + 32, v + 32);
        tmem_wait_ld();
        // pre_p stays fp32 for the tf32 product: release the unit before the stores
        tc_fence_before();
        warp_arrive(&bars->t_full[((c + C::NB) * C::G) % C::NT]);
        uint32_t pk[C::SW / 2];
#pragma unroll
        for (int j = 0; j < C::SW / 2; ++j)
          pk[j] = pack_bf16(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
        // dM_p (bf16) transposed, dMT[(p*H + h) * ld_mt + row], as 4-byte words of two rows: a
        // lane pair swaps its packed (h, h + 1) pairs, then the even lane stores column h of rows
        // (row, row + 1) and the odd lane column h + 1 of rows (row - 1, row)
        const bool odd = lane & 1;
#pragma unroll
        for (int j = 0; j < C::SW / 2; ++j) {
          const uint32_t other = __shfl_xor_sync(0xffffffffu, pk[j], 1);
          const uint32_t word = odd ? __byte_perm(other, pk[j], 0x7632) : __byte_perm(pk[j], other, 0x5410);
          *reinterpret_cast<uint32_t*>(dMT + ((size_t)p * H + C::SW * hh + 2 * j + odd) * ld_mt +
                                       (row & ~1)) = word;
        }
      }
      if (!ok) break;
      if (!mbar_wait(&bars->y_full, i & 1, status, 402, abort, 64)) break;
      tc_fence_after();
      // Y leaves TMEM in groups, each read completely before any global traffic of its own; after
      // the last group's read the next tile may start accumulating.  Up to H = 64 one group, so
      // the release does not wait on the accumulating backward's reads of the previous dE (wider
      // groups at larger H measured slower: 32 columns there)
      constexpr int YG = H <= 64 ? H : 32;
#pragma unroll
      for (int g0 = 0; g0 < H; g0 += YG) {
        uint32_t vg[YG];
        tmem_ld32(tmem + lane_base + C::YCOL + g0, vg);
        if constexpr (YG > 32) tmem_ld32(tmem + lane_base + C::YCOL + g0 + 32, vg + 32);
        tmem_wait_ld();
        if (g0 + YG >= H) {
          tc_fence_before();
          warp_arrive(&bars->y_empty);
        }
        if (asl >= 0) {
          const float* ad = sc.addend + (size_t)asl * H + g0;
#pragma unroll
          for (int j = 0; j < YG; ++j) vg[j] = __float_as_uint(__uint_as_float(vg[j]) + ad[j]);
        }
        if (C::GM && !BWD && sc.bias && part <= 0) {
          // the bias: in-degree of each type (an exact 16-bit integer) times b_p, in fp32
          const uint16_t* dr = sc.deg + (size_t)row * 64;
          for (int q = 0; q < P; ++q) {
            const uint32_t bits = dr[q];
            if (!bits) continue;
            const float d = sc.bias_f16 ? __half2float(__ushort_as_half((unsigned short)bits))
                                        : __uint_as_float(bits << 16);
            const float* bq = sc.bias + (size_t)q * H + g0;
#pragma unroll
            for (int j = 0; j < YG; ++j) vg[j] = __float_as_uint(fmaf(d, bq[j], __uint_as_float(vg[j])));
          }
        }
#pragma unroll
        for (int h1 = 0; h1 < YG; h1 += 32) {
          const int h0 = g0 + h1;
          const uint32_t* v = vg + h1;
          if (part >= 0) {
            // a slice of a split tile: its partial Y, summed with the other slices' by the fix-up
            float4* o = reinterpret_cast<float4*>(
                sc.part + ((size_t)part * sc.part_rows + (size_t)(k - sc.n_full) * kTile + r) * H + h0);
#pragma unroll
            for (int j = 0; j < 8; ++j)
              o[j] = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                 __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
            continue;
          }
          if (out) {
            float4* o = reinterpret_cast<float4*>(out + (size_t)row * H + h0);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              float4 a = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                     __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
              if (accumulate) {
                const float4 prev = o[j];
                a.x += prev.x; a.y += prev.y; a.z += prev.z; a.w += prev.w;
              }
              o[j] = a;
            }
          }
          if (outb || outT) {
            uint32_t pk[16];
#pragma unroll
            for (int j = 0; j < 16; ++j)
              pk[j] = pack_bf16(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
            if (outb) {
              uint4* ob = reinterpret_cast<uint4*>(outb + (size_t)row * H + h0);
#pragma unroll
              for (int j = 0; j < 4; ++j)
                ob[j] = make_uint4(pk[4 * j], pk[4 * j + 1], pk[4 * j + 2], pk[4 * j + 3]);
            }
            if (outT) {
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                __nv_bfloat16* d = outT + (size_t)(h0 + 2 * j) * ld_outT + row;
                d[0] = __ushort_as_bfloat16((unsigned short)(pk[j] & 0xFFFFu));
                d[ld_outT] = __ushort_as_bfloat16((unsigned short)(pk[j] >> 16));
              }
            }
          }
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

// ------------------------------------------------------------------------------------ prep
// out[c][r] = bf16(in[r][c]) for an R x Cc row-major input (batched over blockIdx.z)
template <typename T>
__global__ void k_transpose_bf16(const T* __restrict__ in, __nv_bfloat16* __restrict__ out, int R,
                                 int Cc, int64_t in_batch, int64_t out_batch, int64_t ld_out) {
  __shared__ float tile[32][33];
  in += blockIdx.z * in_batch;
  out += blockIdx.z * out_batch;
  const int r0 = blockIdx.y * 32, c0 = blockIdx.x * 32;
  for (int dy = threadIdx.y; dy < 32; dy += blockDim.y) {
    const int r = r0 + dy, c = c0 + threadIdx.x;
    float v = 0.f;
    if (r < R && c < Cc) {
      if constexpr (sizeof(T) == 2)
        v = __bfloat162float(in[(int64_t)r * Cc + c]);
      else
        v = in[(int64_t)r * Cc + c];
    }
    tile[dy][threadIdx.x] = v;
  }
  __syncthreads();
  for (int dy = threadIdx.y; dy < 32; dy += blockDim.y) {
    const int c = c0 + dy, r = r0 + threadIdx.x;
    if (c < Cc && r < R) out[(int64_t)c * ld_out + r] = __float2bfloat16_rn(tile[threadIdx.x][dy]);
  }
}

// Second-product weights in the band kernel's operand layout, for each type p:
//   forward  out[p][o][i] = W[p][i][o]   (W_p^T, K-major in i)
//   backward out[p][i][o] = W[p][i][o]   (W_p as given, K-major in o)
// as fp32 (the tf32 product's B operand).
__global__ void k_prep_w(const __nv_bfloat16* __restrict__ W, float* __restrict__ out, int P, int H,
                         int transpose) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= (int64_t)P * H * H) return;
  const int64_t p = t / ((int64_t)H * H);
  const int a = (int)((t / H) % H), c = (int)(t % H);
  out[t] = __bfloat162float(transpose ? W[(p * H + c) * H + a] : W[(p * H + a) * H + c]);
}

// Outputs of the split tiles: Y = sum over the ksplit slices of `part` (fixed order), written like
// the band kernel's own epilogue (fp32 out, accumulating if asked; bf16 row-major; bf16
// transposed).  Rows row0 .. row0 + part_rows.
__global__ void k_band_split_fixup(const float* __restrict__ part, int ksplit, int part_rows,
                                   int row0, int H, float* __restrict__ out,
                                   __nv_bfloat16* __restrict__ outb,
                                   __nv_bfloat16* __restrict__ outT, int64_t ld_outT,
                                   int accumulate, const float* __restrict__ addend,
                                   const int32_t* __restrict__ slot) {
  grid_dep_wait();  // the partials are the band kernel's output
  const int64_t n4 = (int64_t)part_rows * H / 4, slice = (int64_t)part_rows * H;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < n4;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t e = 4 * t;
    float4 y = *reinterpret_cast<const float4*>(part + e);
    for (int q = 1; q < ksplit; ++q) {
      const float4 v = *reinterpret_cast<const float4*>(part + q * slice + e);
      y.x += v.x; y.y += v.y; y.z += v.z; y.w += v.w;
    }
    const int row = row0 + (int)(e / H), h = (int)(e % H);
    if (addend && slot[row] >= 0) {
      const float4 a = *reinterpret_cast<const float4*>(addend + (size_t)slot[row] * H + h);
      y.x += a.x; y.y += a.y; y.z += a.z; y.w += a.w;
    }
    if (out) {
      float4* o = reinterpret_cast<float4*>(out + (size_t)row * H + h);
      if (accumulate) {
        const float4 prev = *o;
        y.x += prev.x; y.y += prev.y; y.z += prev.z; y.w += prev.w;
      }
      *o = y;
    }
    const uint32_t p0 = pack_bf16(y.x, y.y), p1 = pack_bf16(y.z, y.w);
    if (outb) *reinterpret_cast<uint2*>(outb + (size_t)row * H + h) = make_uint2(p0, p1);
    if (outT) {
      outT[(size_t)h * ld_outT + row] = __ushort_as_bfloat16((unsigned short)(p0 & 0xFFFFu));
      outT[(size_t)(h + 1) * ld_outT + row] = __ushort_as_bfloat16((unsigned short)(p0 >> 16));
      outT[(size_t)(h + 2) * ld_outT + row] = __ushort_as_bfloat16((unsigned short)(p1 & 0xFFFFu));
      outT[(size_t)(h + 3) * ld_outT + row] = __ushort_as_bfloat16((unsigned short)(p1 >> 16));
    }
  }
}

// b2T[h][p] = high part of b[p][h], b2T[h][32 + p] = the remainder (zero beyond P), both bf16, or
// both fp16 (f16 != 0; the in-degrees are then fp16 too).  fp16 holds magnitudes up to 65504: a
// finite bias beyond that is recorded in the status word (code 2, site 120) and the product is
// then not to be trusted.
__global__ void k_bias_split(const float* __restrict__ b, uint16_t* __restrict__ b2T, int P, int H,
                             int f16, int* status) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= H * 64) return;
  const int h = t / 64, q = t % 64, p = q % 32;
  float x = 0.f;
  if (p < P && b) x = b[p * H + h];
  if (f16) {
    if (fabsf(x) > 65504.f && isfinite(x) && atomicCAS(status, 0, 2) == 0) atomicExch(status + 1, 120);
    const __half hi = __float2half_rn(x);
    b2T[t] = __half_as_ushort(q < 32 ? hi : __float2half_rn(x - __half2float(hi)));
  } else {
    const __nv_bfloat16 hi = __float2bfloat16_rn(x);
    b2T[t] = __bfloat16_as_ushort(q < 32 ? hi : __float2bfloat16_rn(x - __bfloat162float(hi)));
  }
}

// ------------------------------------------------------------------------------------ host
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

bool make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  return make_map_ld(m, base, rows, cols, cols, box_rows);
}

// The W map of the band kernel: fp32 (the tf32 second product), boxes of 32 columns x H rows.
bool make_map_w(CUtensorMap* m, const void* Wk, int P, int H) {
  return make_map_f32(m, Wk, (uint64_t)P * H, H, H);
}

int num_sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

inline size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

// State columns per pass of the band kernel (Cfg::SW) and so its jobs per tile.
int band_jobs(int H, int S, int P) {
  (void)S;
  return H / (H < 64 ? 32 : 64) * P;
}

// Work items of a launch over n_tiles tiles on `sms` SMs, one CTA per SM: whole tiles, and when
// the last round of the grid would be mostly idle, its tiles split over k in {2, 4} job ranges
// (rounds of a k-th of a tile: ceil(k tail / sms) / k).  A split tile costs extra window loads,
// partial-sum traffic and the fix-up launch, measured at about half a tile round, so the split is
// taken only when the tail then lasts less than half a round (single20k: 158 tiles on 152 SMs,
// +28%; a tail of 110 of 152 tiles split four ways measured 9% slower).
Sched make_sched(int n_tiles, int jobs, int sms, bool can_split) {
  Sched sc{};
  sc.n_items = sc.n_full = n_tiles;
  sc.ksplit = 1;
  const int full = (n_tiles / sms) * sms, tail = n_tiles - full;
  if (!can_split || tail == 0) return sc;
  int best = 1;
  double best_t = 1.0;
  for (int k = 2; k <= 4 && k <= jobs; k *= 2) {
    const double t = (double)((k * tail + sms - 1) / sms) / k;
    if (t < best_t - 1e-9) best_t = t, best = k;
  }
  if (best == 1 || best_t >= 0.5) return sc;
  sc.n_full = full;
  sc.ksplit = best;
  sc.n_items = full + best * tail;
  sc.part_rows = tail * kTile;
  return sc;
}

template <int H, int S, bool BWD>
cudaError_t launch_s(const bg_plan* p, const CUtensorMap& tx, const CUtensorMap& tw,
                     const CUtensorMap& tdeg, const CUtensorMap& tb2, float* out,
                     __nv_bfloat16* outb, __nv_bfloat16* outT, int64_t ld_outT,
                     __nv_bfloat16* dMT, int64_t ld_mt, int has_bias, int accumulate,
                     float* split, const float* addend, const float* b32, int* status,
                     cudaStream_t st) {
  using C = Cfg<H, S, BWD>;
  cudaError_t e = cudaFuncSetAttribute(k_band_tc<H, S, BWD>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  const int n_tiles = p->n_pad() / kTile, sms = num_sms();
  Sched sc = make_sched(n_tiles, C::NH * p->P, sms, split != nullptr);
  sc.part = split;
  sc.addend = BWD ? nullptr : addend;
  sc.slot = p->d_sin_slot;
  sc.deg = reinterpret_cast<const uint16_t*>(p->d_deg2);
  sc.bias = (C::GM && !BWD && has_bias) ? b32 : nullptr;
  sc.bias_f16 = p->max_deg > 256 ? 1 : 0;
  const int grid = std::min(sc.n_items, sms);
  e = launch_pdl(k_band_tc<H, S, BWD>, dim3(grid), dim3(C::THREADS), C::SMEM, st, tx, tw, tdeg,
                 tb2, BWD ? p->d_maskTI : p->d_maskI, out, outb, outT, ld_outT, dMT, ld_mt, sc,
                 p->P, has_bias, p->max_deg > 256 ? 1 : 0, accumulate, status);
  note_launch();
  if (e != cudaSuccess || sc.ksplit == 1) return e;
  const int64_t n4 = (int64_t)sc.part_rows * H / 4;
  e = launch_pdl(k_band_split_fixup, dim3((unsigned)std::min<int64_t>((n4 + 255) / 256, 2048)),
                 dim3(256), 0, st, (const float*)split, sc.ksplit, sc.part_rows,
                 sc.n_full * kTile, H, out, outb, outT, ld_outT, accumulate, sc.addend, sc.slot);
  note_launch();
  return e;
}

// The shapes with a tensor-core kernel: H in {32, 64, 128} at S in {32, 64, 128, 256, 512}; H = 256
// at S in {32, 64, 128} (its state-slice window at S = 256 leaves no room for the mask ring).
template <int H, bool BWD>
cudaError_t launch(const bg_plan* p, const CUtensorMap& tx, const CUtensorMap& tw,
                   const CUtensorMap& tdeg, const CUtensorMap& tb2, float* out,
                   __nv_bfloat16* outb, __nv_bfloat16* outT, int64_t ld_outT,
                   __nv_bfloat16* dMT, int64_t ld_mt, int has_bias, int accumulate, float* split,
                   const float* addend, const float* b32, int* status, cudaStream_t st) {
#define BG_BAND_S(SV)                                                                            \
  return launch_s<H, SV, BWD>(p, tx, tw, tdeg, tb2, out, outb, outT, ld_outT, dMT, ld_mt,      \
                              has_bias, accumulate, split, addend, b32, status, st);
  switch (p->S) {
    case 32: BG_BAND_S(32)
    case 64: BG_BAND_S(64)
    case 256:
      if constexpr (H <= 128) { BG_BAND_S(256) }
      return cudaErrorInvalidValue;
    case 512:
      if constexpr (H <= 128) { BG_BAND_S(512) }
      return cudaErrorInvalidValue;
    default: BG_BAND_S(128)
  }
#undef BG_BAND_S
}

}  // namespace

// Row-major fp32 [rows][cols], boxes of 32 columns (one 128-byte swizzle row) x box_rows.
bool make_map_f32(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols,
                  uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 4};
  cuuint32_t box[2] = {32, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool make_map_ld(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint64_t ld,
                 uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int gemm_tn_num_sms() { return num_sms(); }

bool make_map_3d(CUtensorMap* m, const void* base, uint64_t batch, uint64_t rows, uint64_t cols,
                 uint64_t ld, uint64_t sbatch, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {cols, rows, batch};
  cuuint64_t strides[2] = {ld * 2, sbatch * 2};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool band_tc_supported(const bg_plan* p, int dtype, int H) {
  if (!p || dtype != 1 || p->P > 32 || p->n_pad() % kTile) return false;
  const bool shape = ((H == 32 || H == 64 || H == 128) &&
                      (p->S == 32 || p->S == 64 || p->S == 128 || p->S == 256 || p->S == 512)) ||
                     (H == 256 && (p->S == 32 || p->S == 64 || p->S == 128));
  return shape && p->d_maskI && p->d_maskTI && p->d_deg2 && p->max_deg < 2048 &&
         encode_fn() != nullptr;
}

size_t band_tc_w_bytes(const bg_plan* p, int H) {
  return al256((size_t)p->P * H * H * 4);
}

cudaError_t band_tc_prep_w(const bg_plan* p, int H, const void* W, int bwd, void* Wk,
                           cudaStream_t st) {
  const int64_t n = (int64_t)p->P * H * H;
  const int blocks = (int)((n + 255) / 256);
  const auto* w = static_cast<const __nv_bfloat16*>(W);
  k_prep_w<<<blocks, 256, 0, st>>>(w, static_cast<float*>(Wk), p->P, H, !bwd);
  note_launch();
  return cudaGetLastError();
}

size_t band_tc_fwd_ws_bytes(const bg_plan* p, int dtype, int H) {
  if (!p || dtype != 1) return 0;
  const size_t n = (size_t)p->n_pad();
  return al256(n * H * 2) + band_tc_w_bytes(p, H) + al256((size_t)H * 64 * 2) +
         al256(sizeof(float) * band_tc_split_floats(p, H));
}

size_t band_tc_bwd_ws_bytes(const bg_plan* p, int dtype, int H) {
  if (!p || dtype != 1) return 0;
  const size_t n = (size_t)p->n_pad();
  return al256(n * H * 2) + al256((size_t)p->P * H * n * 2) + al256((size_t)(H + 16) * n * 2) +
         band_tc_w_bytes(p, H) +
         al256(sizeof(float) * gemm_tn_part_floats(p->P * H, H + 16, (int64_t)n)) +
         al256(sizeof(float) * band_tc_split_floats(p, H));
}

size_t band_tc_split_floats(const bg_plan* p, int H) {
  const Sched sc = make_sched(p->n_pad() / kTile, band_jobs(H, p->S, p->P), num_sms(), true);
  return sc.ksplit > 1 ? (size_t)sc.ksplit * sc.part_rows * H : 0;
}

cudaError_t band_tc_fwd_core(const bg_plan* p, int H, const __nv_bfloat16* XT, int64_t ld_x,
                             const void* Wk, const __nv_bfloat16* b2T, const float* b32,
                             float* out, __nv_bfloat16* outb, __nv_bfloat16* outT,
                             int64_t ld_outT, float* split, const float* addend, int* status,
                             cudaStream_t st) {
  const int n = p->n_pad(), P = p->P;
  CUtensorMap tx, tw, tdeg, tb2;
  if (!make_map_ld(&tx, XT, H, n, ld_x, H < 64 ? 32 : 64) ||
      !make_map_w(&tw, Wk, P, H) || !make_map(&tdeg, p->d_deg2, n, 64, kTile) ||
      !make_map(&tb2, b2T ? b2T : XT, H, 64, H))
    return cudaErrorInvalidValue;
  const int hb = b2T != nullptr;
#define BG_FWD(HV)                                                                                \
  return launch<HV, false>(p, tx, tw, tdeg, tb2, out, outb, outT, ld_outT, nullptr, 0, hb, 0,     \
                           split, addend, b32, status, st);
  switch (H) {
    case 32: BG_FWD(32)
    case 64: BG_FWD(64)
    case 128: BG_FWD(128)
    default: BG_FWD(256)
  }
#undef BG_FWD
}

cudaError_t band_tc_bwd_core(const bg_plan* p, int H, const __nv_bfloat16* dYT, int64_t ld_y,
                             const void* Wk, float* dE, int accumulate, __nv_bfloat16* dMT,
                             int64_t ld_mt, float* split, int* status, cudaStream_t st) {
  const int n = p->n_pad(), P = p->P;
  CUtensorMap tx, tw;
  if (!make_map_ld(&tx, dYT, H, n, ld_y, H < 64 ? 32 : 64) ||
      !make_map_w(&tw, Wk, P, H))
    return cudaErrorInvalidValue;
#define BG_BWD(HV)                                                                                \
  return launch<HV, true>(p, tx, tw, tw, tw, dE, nullptr, nullptr, 0, dMT, ld_mt, 0, accumulate,  \
                          split, nullptr, nullptr, status, st);
  switch (H) {
    case 32: BG_BWD(32)
    case 64: BG_BWD(64)
    case 128: BG_BWD(128)
    default: BG_BWD(256)
  }
#undef BG_BWD
}

cudaError_t prep_transpose_bf16(const void* in, int in_is_f32, __nv_bfloat16* out, int R, int Cc,
                                int batch, cudaStream_t st, int64_t ld_out) {
  dim3 grid((Cc + 31) / 32, (R + 31) / 32, batch);
  if (ld_out <= 0) ld_out = R;
  if (in_is_f32)
    k_transpose_bf16<float><<<grid, dim3(32, 8), 0, st>>>(static_cast<const float*>(in), out, R, Cc,
                                                          (int64_t)R * Cc, (int64_t)R * Cc, ld_out);
  else
    k_transpose_bf16<__nv_bfloat16><<<grid, dim3(32, 8), 0, st>>>(
        static_cast<const __nv_bfloat16*>(in), out, R, Cc, (int64_t)R * Cc, (int64_t)R * Cc,
        ld_out);
  note_launch();
  return cudaGetLastError();
}

cudaError_t prep_bias_split(const bg_plan* p, const float* b, __nv_bfloat16* b2T, int H,
                            int* status, cudaStream_t st) {
  k_bias_split<<<(H * 64 + 255) / 256, 256, 0, st>>>(b, reinterpret_cast<uint16_t*>(b2T), p->P, H,
                                                     p->max_deg > 256 ? 1 : 0, status);
  note_launch();
  return cudaGetLastError();
}

cudaError_t band_tc_fwd(const bg_plan* p, int H, const void* E, const void* W, const float* b,
                        float* Y, char* ws, size_t ws_bytes, int* status, cudaStream_t st) {
  if (ws_bytes < band_tc_fwd_ws_bytes(p, 1, H)) return cudaErrorInvalidValue;
  const int n = p->n_pad();
  __nv_bfloat16* ET = reinterpret_cast<__nv_bfloat16*>(ws);
  void* WT = ws + al256((size_t)n * H * 2);
  __nv_bfloat16* b2T = reinterpret_cast<__nv_bfloat16*>(ws + al256((size_t)n * H * 2) +
                                                        band_tc_w_bytes(p, H));
  float* split = reinterpret_cast<float*>(ws + al256((size_t)n * H * 2) + band_tc_w_bytes(p, H) +
                                          al256((size_t)H * 64 * 2));
  // E [n][H] -> ET [H][n];  W_p [H_in][H_out] -> W_p^T in the kernel's operand type;  bias split
  cudaError_t e = prep_transpose_bf16(E, 0, ET, n, H, 1, st);
  if (e == cudaSuccess) e = band_tc_prep_w(p, H, W, 0, WT, st);
  if (e == cudaSuccess && b) e = prep_bias_split(p, b, b2T, H, status, st);
  if (e != cudaSuccess) return e;
  ProfSpan span(BG_KID_BAND_FWD, st);
  return band_tc_fwd_core(p, H, ET, n, WT, b ? b2T : nullptr, b, Y, nullptr, nullptr, 0,
                          band_tc_split_floats(p, H) ? split : nullptr, nullptr, status, st);
}

cudaError_t band_tc_bwd(const bg_plan* p, int H, const void* E, const void* W, const float* dY,
                        float* dE, float* dW, float* db, int accum, char* ws, size_t ws_bytes,
                        int* status, cudaStream_t st) {
  if (ws_bytes < band_tc_bwd_ws_bytes(p, 1, H)) return cudaErrorInvalidValue;
  const int n = p->n_pad(), P = p->P;
  size_t o = 0;
  __nv_bfloat16* dYT = reinterpret_cast<__nv_bfloat16*>(ws + o);
  o += al256((size_t)n * H * 2);
  __nv_bfloat16* dMT = reinterpret_cast<__nv_bfloat16*>(ws + o);
  o += al256((size_t)P * H * n * 2);
  __nv_bfloat16* ETa = reinterpret_cast<__nv_bfloat16*>(ws + o);
  o += al256((size_t)(H + 16) * n * 2);
  void* Wk = ws + o;
  o += band_tc_w_bytes(p, H);
  float* part = reinterpret_cast<float*>(ws + o);
  const size_t part_floats = gemm_tn_part_floats(P * H, H + 16, (int64_t)n);
  o += al256(sizeof(float) * part_floats);
  float* split = band_tc_split_floats(p, H) ? reinterpret_cast<float*>(ws + o) : nullptr;
  cudaError_t e = prep_transpose_bf16(dY, 1, dYT, n, H, 1, st);
  if (e == cudaSuccess) e = band_tc_prep_w(p, H, W, 1, Wk, st);
  if (e == cudaSuccess) {
    ProfSpan span(BG_KID_BAND_BWD, st);
    e = band_tc_bwd_core(p, H, dYT, n, Wk, dE, accum, dMT, n, split, status, st);
  }
  if (e != cudaSuccess) return e;
  // E^T; the weight-gradient product appends its ones row, which turns the bias gradient into
  // column H of the same product
  e = prep_transpose_bf16(E, 0, ETa, n, H, 1, st);
  if (e != cudaSuccess) return e;
  // dW_p[h][h'] (+)= sum_nodes E[node][h] dM_p[node][h'],  db_p[h'] (+)= sum_nodes dM_p[node][h']
  ProfSpan span(BG_KID_DW, st);
  return gemm_tn(dMT, n, ETa, n, P * H, H, n, 1, dW, db, accum, part, part_floats, status, st);
}

int band_tc_upload(bg_plan* p, cudaStream_t st) {
  const int S = p->S;
  if (p->P > 32 || (S != 32 && S != 64 && S != 128 && S != 256 && S != 512)) return 0;
  const size_t n = (size_t)p->K * S;
  if (n % kTile) return 0;
  std::vector<uint32_t> mi, mti;
  std::vector<uint16_t> deg;
  const int max_deg = band_tc_host_tiles(p, band_chunks(S), mi, mti, deg);
  p->max_deg = max_deg;
  if (cudaMalloc(&p->d_maskI, mi.size() * 4) != cudaSuccess ||
      cudaMalloc(&p->d_maskTI, mti.size() * 4) != cudaSuccess ||
      cudaMalloc(&p->d_deg2, deg.size() * 2) != cudaSuccess)
    return -1;
  if (cudaMemcpyAsync(p->d_maskI, mi.data(), mi.size() * 4, cudaMemcpyHostToDevice, st) != cudaSuccess ||
      cudaMemcpyAsync(p->d_maskTI, mti.data(), mti.size() * 4, cudaMemcpyHostToDevice, st) != cudaSuccess ||
      cudaMemcpyAsync(p->d_deg2, deg.data(), deg.size() * 2, cudaMemcpyHostToDevice, st) != cudaSuccess)
    return -1;
  if (cudaStreamSynchronize(st) != cudaSuccess) return -1;
  return 0;
}

cudaError_t band_tc_preload_fwd(const bg_plan* p) {
  if (!encode_fn()) return cudaErrorNotSupported;
  cudaFuncAttributes a;
  cudaError_t e = cudaSuccess;
  auto take = [&](cudaError_t r) { if (e == cudaSuccess) e = r; };
  take(cudaFuncGetAttributes(&a, k_transpose_bf16<__nv_bfloat16>));
  take(cudaFuncGetAttributes(&a, k_prep_w));
  take(cudaFuncGetAttributes(&a, k_bias_split));
  take(cudaFuncGetAttributes(&a, k_band_split_fixup));
#define BG_PRELOAD(HV, SV) take(cudaFuncGetAttributes(&a, k_band_tc<HV, SV, false>));
#define BG_PRELOAD_S(SV) BG_PRELOAD(32, SV) BG_PRELOAD(64, SV) BG_PRELOAD(128, SV)
  switch (p->S) {
    case 32: BG_PRELOAD_S(32) BG_PRELOAD(256, 32) break;
    case 64: BG_PRELOAD_S(64) BG_PRELOAD(256, 64) break;
    case 128: BG_PRELOAD_S(128) BG_PRELOAD(256, 128) break;
    case 256: BG_PRELOAD_S(256) break;
    case 512: BG_PRELOAD_S(512) break;
    default: break;
  }
#undef BG_PRELOAD_S
#undef BG_PRELOAD
  return e;
}

void band_tc_release(bg_plan* p) {
  cudaFree(p->d_maskI);
  cudaFree(p->d_maskTI);
  cudaFree(p->d_deg2);
  p->d_maskI = p->d_maskTI = nullptr;
  p->d_deg2 = nullptr;
}

}  // namespace bg

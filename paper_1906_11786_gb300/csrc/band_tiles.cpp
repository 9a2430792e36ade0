// Host side of the tensor-core path's plan data (band_tc.cu uploads what this builds).
//
// For every 128-row tile and edge type: the C1 128-column chunks of the tile's state window
// [ws, ws + 128 C1), ws = (row0 / S) S - S, as 4 words per row and chunk, in both orientations,
// with the bits of each word interleaved (column 2j at bit j, column 2j+1 at bit 16+j) so that the
// kernel turns a word into packed bf16 pairs with one AND and one multiply; words outside the three
// block diagonals of the row's block-row are zero.  And per row and type the in-degree over the
// three diagonals (columns p and 32 + p), the bias product's A operand: bf16 integers when every
// in-degree is at most 256, fp16 integers otherwise (a hub node; fp16 is exact up to 2048).
#include <algorithm>
#include <cstring>
#include <thread>
#include <vector>

#include "band_tc.h"
#include "internal.h"

namespace bg {

namespace {

// Bits 0, 2, 4, ... of x packed into bits 0..15 (even-bit compaction by shifts and masks).
inline uint32_t even_bits(uint32_t x) {
  x &= 0x55555555u;
  x = (x | (x >> 1)) & 0x33333333u;
  x = (x | (x >> 2)) & 0x0F0F0F0Fu;
  x = (x | (x >> 4)) & 0x00FF00FFu;
  x = (x | (x >> 8)) & 0x0000FFFFu;
  return x;
}

// Column 2j -> bit j, column 2j+1 -> bit 16+j.
inline uint32_t interleave(uint32_t w) {
  return w == 0 ? 0u : even_bits(w) | (even_bits(w >> 1) << 16);
}

// Runs f(lo, hi) over [0, n) split into contiguous ranges on up to 16 host threads.
template <typename F>
void parallel_ranges(int64_t n, F f) {
  unsigned nt = std::max(1u, std::min(std::thread::hardware_concurrency(), 16u));
  if ((int64_t)nt > n) nt = (unsigned)std::max<int64_t>(1, n);
  std::vector<std::thread> pool;
  for (unsigned t = 1; t < nt; ++t)
    pool.emplace_back([=]() { f(n * t / nt, n * (t + 1) / nt); });
  f(0, n / nt);
  for (auto& th : pool) th.join();
}

// bf16 bit pattern of a count (exact up to 256).
inline uint16_t bf16_bits_of_count(int c) {
  const float f = (float)c;
  uint32_t u;
  std::memcpy(&u, &f, 4);
  return (uint16_t)(u >> 16);
}

// IEEE fp16 bit pattern of a count in [0, 2048) (exact: at most 11 significant bits).
inline uint16_t f16_bits_of_count(int c) {
  if (c == 0) return 0;
  int e = 0;
  while ((c >> (e + 1)) != 0) ++e;  // floor(log2 c)
  const uint32_t mant = ((uint32_t)c << (10 - e)) & 0x3FFu;
  return (uint16_t)(((uint32_t)(e + 15) << 10) | mant);
}

}  // namespace

// mi, mti: [n_tiles][P][C1][128][4] words; deg: [n_pad][64] in-degrees (type q at columns q and
// 32 + q) as bf16 when the largest is at most 256, else as fp16.  Returns the largest in-degree.
int band_tc_host_tiles(const bg_plan* p, int C1, std::vector<uint32_t>& mi,
                       std::vector<uint32_t>& mti, std::vector<uint16_t>& deg) {
  constexpr int kTile = 128;
  const int S = p->S, K = p->K, P = p->P, W32 = p->W32;
  const int64_t n = (int64_t)K * S, n_tiles = n / kTile;
  mi.assign((size_t)n_tiles * P * C1 * kTile * 4, 0u);
  mti.assign(mi.size(), 0u);
  deg.assign((size_t)n * 64, 0);
  parallel_ranges(n_tiles, [&](int64_t t0, int64_t t1) {
    for (int64_t t = t0; t < t1; ++t) {
      const int64_t row0 = t * kTile, ws = (row0 / S) * S - S;
      for (int q = 0; q < P; ++q)
        for (int j = 0; j < C1; ++j)
          for (int r = 0; r < kTile; ++r)
            for (int w = 0; w < 4; ++w) {
              const int64_t R = row0 + r, Cc = ws + j * kTile + 32 * w;
              if (Cc < 0 || Cc >= n) continue;
              const int64_t kr = R / S, kc = Cc / S, d = kc - kr + 1;
              if (d < 0 || d > 2) continue;
              const size_t dst = ((((size_t)t * P + q) * C1 + j) * kTile + r) * 4 + w;
              const size_t src = ((((size_t)kr * 3 + d) * P + q) * S + R % S) * W32 + (Cc % S) / 32;
              mi[dst] = interleave(p->masks[src]);
              mti[dst] = interleave(p->masksT[src]);
            }
    }
  });
  // in-degrees first, then their encoding: bf16 while every count is at most 256 (exact), else
  // fp16 (exact up to 2048 > 3 S for every block size)
  std::vector<uint16_t> cnt((size_t)n * P, 0);
  std::vector<int> part_max(K, 0);
  parallel_ranges(K, [&](int64_t k0, int64_t k1) {
    for (int64_t k = k0; k < k1; ++k) {
      int mx = 0;
      for (int q = 0; q < P; ++q)
        for (int r = 0; r < S; ++r) {
          int c = 0;
          for (int d = 0; d < 3; ++d)
            for (int w = 0; w < W32; ++w)
              c += __builtin_popcount(p->masks[((((size_t)k * 3 + d) * P + q) * S + r) * W32 + w]);
          mx = std::max(mx, c);
          cnt[((size_t)k * S + r) * P + q] = (uint16_t)c;
        }
      part_max[k] = mx;
    }
  });
  const int max_deg = *std::max_element(part_max.begin(), part_max.end());
  const bool f16 = max_deg > 256;
  parallel_ranges(n, [&](int64_t r0, int64_t r1) {
    for (int64_t r = r0; r < r1; ++r)
      for (int q = 0; q < P; ++q) {
        const uint16_t v = f16 ? f16_bits_of_count(cnt[(size_t)r * P + q])
                               : bf16_bits_of_count(cnt[(size_t)r * P + q]);
        deg[(size_t)r * 64 + q] = v;
        deg[(size_t)r * 64 + 32 + q] = v;
      }
  });
  return max_deg;
}

}  // namespace bg

// Test helper for tests/test_plan_abi.py: plans the graphs of a binary file and writes the plan's
// forward bit tiles together with the host-built operands of the tensor-core path (window chunks
// of interleaved bits in both orientations, per-row in-degrees as bf16), so that the test can
// rebuild the latter from the former on its own.
//
//   tiles_probe IN OUT P S C1
//   IN:  int32 n_graphs, then per graph int32 n_nodes, int64 n_edges, int32 src[], dst[], etype[]
//   OUT: int32 K, int32 max_deg, int64 word counts (masks, maskI, maskTI, deg), then the arrays
#include <cstdio>
#include <cstdlib>
#include <vector>

#include "internal.h"

namespace bg {
int band_tc_host_tiles(const bg_plan* p, int C1, std::vector<uint32_t>& mi,
                       std::vector<uint32_t>& mti, std::vector<uint16_t>& deg);
}

int main(int argc, char** argv) {
  if (argc != 6) return 2;
  const int P = std::atoi(argv[3]), S = std::atoi(argv[4]), C1 = std::atoi(argv[5]);
  FILE* f = std::fopen(argv[1], "rb");
  if (!f) return 3;
  int32_t ng = 0;
  if (std::fread(&ng, 4, 1, f) != 1 || ng < 1) return 4;
  std::vector<std::vector<int32_t>> src(ng), dst(ng), et(ng);
  std::vector<bg_graph> gs(ng);
  for (int g = 0; g < ng; ++g) {
    int32_t n = 0;
    int64_t m = 0;
    if (std::fread(&n, 4, 1, f) != 1 || std::fread(&m, 8, 1, f) != 1 || m < 0) return 5;
    src[g].resize(m); dst[g].resize(m); et[g].resize(m);
    if (m && (std::fread(src[g].data(), 4, m, f) != (size_t)m ||
              std::fread(dst[g].data(), 4, m, f) != (size_t)m ||
              std::fread(et[g].data(), 4, m, f) != (size_t)m))
      return 6;
    gs[g] = bg_graph{n, m, src[g].data(), dst[g].data(), et[g].data()};
  }
  std::fclose(f);
  bg_plan* pl = nullptr;
  if (bg_band_plan(gs.data(), ng, P, S, 0, BG_RCM | BG_KEEP_IF_BETTER, &pl) != BG_OK) return 7;
  std::vector<uint32_t> mi, mti;
  std::vector<uint16_t> deg;
  const int32_t max_deg = bg::band_tc_host_tiles(pl, C1, mi, mti, deg);
  FILE* o = std::fopen(argv[2], "wb");
  if (!o) return 8;
  const int32_t K = pl->K;
  const int64_t counts[4] = {(int64_t)pl->masks.size(), (int64_t)mi.size(), (int64_t)mti.size(),
                             (int64_t)deg.size()};
  std::fwrite(&K, 4, 1, o);
  std::fwrite(&max_deg, 4, 1, o);
  std::fwrite(counts, 8, 4, o);
  std::fwrite(pl->masks.data(), 4, pl->masks.size(), o);
  std::fwrite(pl->masksT.data(), 4, pl->masksT.size(), o);
  std::fwrite(mi.data(), 4, mi.size(), o);
  std::fwrite(mti.data(), 4, mti.size(), o);
  std::fwrite(deg.data(), 2, deg.size(), o);
  std::fclose(o);
  bg_plan_free(pl);
  return 0;
}

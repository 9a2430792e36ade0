// Reachability preprocessing (Section 4 "Reachability preprocessing"), host side.
//
// With T propagation steps a node's initial state reaches exactly the nodes within T directed
// hops of it, so only nodes from which some candidate node is reachable in at most T steps can
// change the candidates' final states; the rest of the graph is discarded before planning.  The
// distances come from one breadth-first search that starts at all candidates at once and walks
// the edges backwards (CSR of in-edges), stopping at depth T.
#include <cstring>
#include <string>
#include <vector>

#include "internal.h"

extern "C" int bg_reach_filter(const bg_graph* g, const int32_t* cand, int32_t n_cand, int32_t T,
                               int32_t* node_map, int32_t* n_nodes_out, int64_t* n_edges_out,
                               int32_t* src_out, int32_t* dst_out, int32_t* etype_out) {
  bg_clear_error();
  if (!g || !node_map || !n_nodes_out || !n_edges_out) return bg_fail(BG_EINVAL, "NULL argument");
  const int32_t n = g->n_nodes;
  const int64_t m = g->n_edges;
  if (n < 0 || m < 0 || T < 0 || n_cand < 0) return bg_fail(BG_EINVAL, "negative size or T");
  if (m > 0 && (!g->src || !g->dst)) return bg_fail(BG_EINVAL, "NULL edge arrays");
  if (n_cand > 0 && !cand) return bg_fail(BG_EINVAL, "NULL candidates");
  for (int64_t e = 0; e < m; ++e)
    if (g->src[e] < 0 || g->src[e] >= n || g->dst[e] < 0 || g->dst[e] >= n)
      return bg_fail(BG_EINVAL, "edge " + std::to_string(e) + " has a node id out of range");
  // in-edge CSR: for every target, the sources of its edges
  std::vector<int64_t> start((size_t)n + 1, 0);
  for (int64_t e = 0; e < m; ++e) ++start[(size_t)g->dst[e] + 1];
  for (int32_t v = 0; v < n; ++v) start[v + 1] += start[v];
  std::vector<int32_t> srcs((size_t)m);
  {
    std::vector<int64_t> fill(start.begin(), start.end() - 1);
    for (int64_t e = 0; e < m; ++e) srcs[(size_t)fill[g->dst[e]]++] = g->src[e];
  }
  std::vector<int32_t> dist((size_t)n, -1), frontier, next;
  for (int32_t i = 0; i < n_cand; ++i) {
    const int32_t c = cand[i];
    if (c < 0 || c >= n) return bg_fail(BG_EINVAL, "candidate id out of range");
    if (dist[c] < 0) {
      dist[c] = 0;
      frontier.push_back(c);
    }
  }
  for (int32_t d = 1; d <= T && !frontier.empty(); ++d) {
    next.clear();
    for (int32_t v : frontier)
      for (int64_t i = start[v]; i < start[v + 1]; ++i) {
        const int32_t u = srcs[(size_t)i];
        if (dist[u] < 0) {
          dist[u] = d;
          next.push_back(u);
        }
      }
    frontier.swap(next);
  }
  int32_t kept = 0;
  for (int32_t v = 0; v < n; ++v) node_map[v] = dist[v] >= 0 ? kept++ : -1;
  *n_nodes_out = kept;
  int64_t me = 0;
  for (int64_t e = 0; e < m; ++e) {
    const int32_t a = node_map[g->src[e]], b = node_map[g->dst[e]];
    if (a < 0 || b < 0) continue;
    if (src_out) src_out[me] = a;
    if (dst_out) dst_out[me] = b;
    if (etype_out && g->etype) etype_out[me] = g->etype[e];
    ++me;
  }
  *n_edges_out = me;
  return BG_OK;
}

// Host-side compile step (Section 3.1, Section 2 "Sparse batching", Eq. 3).
//
// Per graph: a symmetric CSR neighbourhood, Reverse Cuthill-McKee with a George-Liu
// pseudo-peripheral start (ties broken by (degree, id); components in discovery order; the whole
// sequence reversed), keep-if-better against the input order.  Graphs are reordered in parallel
// on host threads.  Then contiguous packing in input order up to the first graph that does not
// fit, edge deduplication, and the bit-packed S x S tiles of the three block diagonals per edge
// type in both orientations (forward: rows = targets; transposed: rows = sources).
#include <algorithm>
#include <atomic>
#include <cstring>
#include <thread>

#include "internal.h"

namespace {

struct Csr {
  std::vector<int64_t> start;  // n + 1
  std::vector<int32_t> nbr;    // sorted, unique, no self loops
  int32_t deg(int32_t v) const { return (int32_t)(start[v + 1] - start[v]); }
};

Csr build_csr(int32_t n, int64_t m, const int32_t* src, const int32_t* dst) {
  std::vector<int64_t> cnt(n + 1, 0);
  for (int64_t e = 0; e < m; ++e)
    if (src[e] != dst[e]) { ++cnt[src[e] + 1]; ++cnt[dst[e] + 1]; }
  for (int32_t v = 0; v < n; ++v) cnt[v + 1] += cnt[v];
  std::vector<int32_t> raw(cnt[n]);
  std::vector<int64_t> fill(cnt.begin(), cnt.end() - 1);
  for (int64_t e = 0; e < m; ++e) {
    int32_t a = src[e], b = dst[e];
    if (a == b) continue;
    raw[fill[a]++] = b;
    raw[fill[b]++] = a;
  }
  Csr g;
  g.start.assign(n + 1, 0);
  g.nbr.reserve(raw.size());
  for (int32_t v = 0; v < n; ++v) {
    auto b = raw.begin() + cnt[v], e = raw.begin() + cnt[v + 1];
    std::sort(b, e);
    auto last = std::unique(b, e);
    g.nbr.insert(g.nbr.end(), b, last);
    g.start[v + 1] = (int64_t)g.nbr.size();
  }
  return g;
}

// Key that orders nodes by (degree, id).
inline uint64_t deg_id_key(const Csr& g, int32_t v) {
  return ((uint64_t)(uint32_t)g.deg(v) << 32) | (uint32_t)v;
}

// BFS from r: returns the number of levels and the last level's least-(degree, id) node.
// `mark` / `stamp` avoid clearing a visited array per search.
std::pair<int32_t, int32_t> bfs_depth(const Csr& g, int32_t r, std::vector<uint32_t>& mark,
                                      uint32_t stamp, std::vector<int32_t>& q) {
  q.clear();
  q.push_back(r);
  mark[r] = stamp;
  size_t lvl_begin = 0;
  int32_t depth = 0;
  int32_t best = r;
  while (lvl_begin < q.size()) {
    size_t lvl_end = q.size();
    ++depth;
    best = q[lvl_begin];
    for (size_t i = lvl_begin; i < lvl_end; ++i) {
      int32_t u = q[i];
      if (deg_id_key(g, u) < deg_id_key(g, best)) best = u;
      for (int64_t a = g.start[u]; a < g.start[u + 1]; ++a) {
        int32_t v = g.nbr[a];
        if (mark[v] != stamp) { mark[v] = stamp; q.push_back(v); }
      }
    }
    lvl_begin = lvl_end;
  }
  return {depth, best};
}

int64_t bandwidth_of(int64_t m, const int32_t* src, const int32_t* dst, const int32_t* pos) {
  int64_t bw = 0;
  for (int64_t e = 0; e < m; ++e) {
    int64_t a = pos ? pos[src[e]] : src[e];
    int64_t b = pos ? pos[dst[e]] : dst[e];
    bw = std::max(bw, a > b ? a - b : b - a);
  }
  return bw;
}

// perm[new] = old
void reverse_cuthill_mckee(int32_t n, int64_t m, const int32_t* src, const int32_t* dst,
                           bool keep_if_better, int32_t* perm) {
  Csr g = build_csr(n, m, src, dst);
  // candidates for component starts, by (degree, id)
  std::vector<int32_t> by_key(n);
  for (int32_t v = 0; v < n; ++v) by_key[v] = v;
  std::sort(by_key.begin(), by_key.end(),
            [&](int32_t a, int32_t b) { return deg_id_key(g, a) < deg_id_key(g, b); });
  std::vector<uint32_t> mark(n, 0);
  std::vector<char> done(n, 0);
  std::vector<int32_t> q, out;
  out.reserve(n);
  std::vector<uint64_t> keys;
  uint32_t stamp = 0;
  size_t cursor = 0;
  while ((int32_t)out.size() < n) {
    while (done[by_key[cursor]]) ++cursor;
    int32_t r = by_key[cursor];
    auto cur = bfs_depth(g, r, mark, ++stamp, q);
    for (;;) {
      auto nx = bfs_depth(g, cur.second, mark, ++stamp, q);
      if (nx.first > cur.first) { r = cur.second; cur = nx; } else break;
    }
    // Cuthill-McKee numbering from r
    size_t head = out.size();
    out.push_back(r);
    done[r] = 1;
    while (head < out.size()) {
      int32_t u = out[head++];
      keys.clear();
      for (int64_t a = g.start[u]; a < g.start[u + 1]; ++a)
        if (!done[g.nbr[a]]) keys.push_back(deg_id_key(g, g.nbr[a]));
      std::sort(keys.begin(), keys.end());
      for (uint64_t k : keys) {
        int32_t v = (int32_t)(uint32_t)k;
        done[v] = 1;
        out.push_back(v);
      }
    }
  }
  for (int32_t i = 0; i < n; ++i) perm[i] = out[n - 1 - i];
  if (keep_if_better) {
    std::vector<int32_t> pos(n);
    for (int32_t i = 0; i < n; ++i) pos[perm[i]] = i;
    if (bandwidth_of(m, src, dst, pos.data()) > bandwidth_of(m, src, dst, nullptr))
      for (int32_t i = 0; i < n; ++i) perm[i] = i;
  }
}

}  // namespace

int bg_plan_build(const bg_graph* graphs, int32_t n_graphs, int32_t P, int32_t S, int32_t cap,
                  uint32_t flags, int32_t super_min_degree, int32_t max_super, bg_plan** out) {
  if (!out) return bg_fail(BG_EINVAL, "out is NULL");
  *out = nullptr;
  if (n_graphs < 1 || (!graphs)) return bg_fail(BG_EINVAL, "need at least one graph");
  if (!(S == 32 || S == 64 || S == 128 || S == 256 || S == 512))
    return bg_fail(BG_EINVAL, "block size S must be one of 32, 64, 128, 256, 512");
  if (P < 1 || P > 64) return bg_fail(BG_EINVAL, "n_types must be in [1, 64]");
  if (cap < 0) return bg_fail(BG_EINVAL, "capacity_blocks must be >= 0");
  const bool supernodes = (flags & BG_SUPERNODES) != 0;
  if (supernodes && (super_min_degree < 1 || max_super < 0))
    return bg_fail(BG_EINVAL, "supernodes need supernode_min_degree >= 1 and max_supernodes >= 0");
  for (int32_t g = 0; g < n_graphs; ++g) {
    const bg_graph& gr = graphs[g];
    if (gr.n_nodes < 0 || gr.n_edges < 0)
      return bg_fail(BG_EINVAL, "graph " + std::to_string(g) + ": negative count");
    if (gr.n_edges > 0 && (!gr.src || !gr.dst || !gr.etype))
      return bg_fail(BG_EINVAL, "graph " + std::to_string(g) + ": NULL edge array");
    for (int64_t e = 0; e < gr.n_edges; ++e) {
      if (gr.src[e] < 0 || gr.src[e] >= gr.n_nodes || gr.dst[e] < 0 || gr.dst[e] >= gr.n_nodes)
        return bg_fail(BG_EINVAL, "graph " + std::to_string(g) + ": node id out of range");
      if (gr.etype[e] < 0 || gr.etype[e] >= P)
        return bg_fail(BG_EINVAL, "graph " + std::to_string(g) + ": edge type out of range");
    }
  }
  bg_plan* pl = new (std::nothrow) bg_plan();
  if (!pl) return bg_fail(BG_ENOMEM, "host allocation failed");
  pl->S = S; pl->P = P; pl->W32 = S / 32; pl->n_graphs = n_graphs;
  pl->n_nodes.resize(n_graphs);
  pl->node_base.resize(n_graphs + 1, 0);
  int64_t total = 0;
  for (int32_t g = 0; g < n_graphs; ++g) {
    pl->n_nodes[g] = graphs[g].n_nodes;
    pl->node_base[g] = total;
    total += graphs[g].n_nodes;
  }
  pl->node_base[n_graphs] = total;
  int64_t K64 = cap > 0 ? cap : (total + S - 1) / S;
  if (K64 < 1) K64 = 1;
  if (K64 * S > ((int64_t)1 << 28)) { delete pl; return bg_fail(BG_EINVAL, "supergraph too large"); }
  pl->K = (int32_t)K64;
  const int64_t capacity = K64 * S;

  // packing decision (depends only on node counts, Section 2 "Sparse batching")
  pl->offset.assign(n_graphs, -1);
  int64_t pos = 0;
  for (int32_t g = 0; g < n_graphs; ++g) {
    if (pos + graphs[g].n_nodes > capacity) break;
    pl->offset[g] = (int32_t)pos;
    pos += graphs[g].n_nodes;
    ++pl->n_packed;
  }
  if (pl->n_packed == 0) { delete pl; return bg_fail(BG_ECAPACITY, "first graph exceeds the capacity"); }
  pl->n_real = (int32_t)pos;

  // reorder every input graph (identity where RCM is off) so that the exported permutation
  // covers all of them; threads take graphs from a shared counter
  pl->perm.resize(total);
  pl->bw_before.assign(n_graphs, 0);
  pl->bw_after.assign(n_graphs, 0);
  pl->nsup.assign(n_graphs, 0);
  std::atomic<int32_t> next{0};
  auto worker = [&]() {
    for (;;) {
      int32_t g = next.fetch_add(1);
      if (g >= n_graphs) return;
      const bg_graph& gr = graphs[g];
      const int32_t n = gr.n_nodes;
      int32_t* pg = pl->perm.data() + pl->node_base[g];
      // supernodes: degree (distinct neighbours, self-loops not counted) at least the threshold,
      // highest degree first, ties by id, at most max_super; they take the first positions
      std::vector<int32_t> sup;
      if (supernodes && max_super > 0) {
        Csr c = build_csr(n, gr.n_edges, gr.src, gr.dst);
        for (int32_t v = 0; v < n; ++v)
          if (c.deg(v) >= super_min_degree) sup.push_back(v);
        std::sort(sup.begin(), sup.end(), [&](int32_t a, int32_t b) {
          return c.deg(a) != c.deg(b) ? c.deg(a) > c.deg(b) : a < b;
        });
        if ((int32_t)sup.size() > max_super) sup.resize(max_super);
      }
      pl->nsup[g] = (int32_t)sup.size();
      std::vector<char> is_sup(n, 0);
      for (int32_t v : sup) is_sup[v] = 1;
      if (sup.empty()) {
        if (flags & BG_RCM) {
          reverse_cuthill_mckee(n, gr.n_edges, gr.src, gr.dst, (flags & BG_KEEP_IF_BETTER) != 0, pg);
        } else {
          for (int32_t i = 0; i < n; ++i) pg[i] = i;
        }
      } else {
        // the graph without its supernodes, renumbered in ascending id, ordered on its own
        std::vector<int32_t> rest, rid(n, -1), rs, rd;
        for (int32_t v = 0; v < n; ++v)
          if (!is_sup[v]) { rid[v] = (int32_t)rest.size(); rest.push_back(v); }
        for (int64_t e = 0; e < gr.n_edges; ++e)
          if (!is_sup[gr.src[e]] && !is_sup[gr.dst[e]]) { rs.push_back(rid[gr.src[e]]); rd.push_back(rid[gr.dst[e]]); }
        const int32_t nr = (int32_t)rest.size();
        std::vector<int32_t> pr(nr);
        if (flags & BG_RCM) {
          reverse_cuthill_mckee(nr, (int64_t)rs.size(), rs.data(), rd.data(),
                                (flags & BG_KEEP_IF_BETTER) != 0, pr.data());
        } else {
          for (int32_t i = 0; i < nr; ++i) pr[i] = i;
        }
        for (size_t i = 0; i < sup.size(); ++i) pg[i] = sup[i];
        for (int32_t i = 0; i < nr; ++i) pg[sup.size() + i] = rest[pr[i]];
      }
      std::vector<int32_t> where(n);
      for (int32_t i = 0; i < n; ++i) where[pg[i]] = i;
      pl->bw_before[g] = bandwidth_of(gr.n_edges, gr.src, gr.dst, nullptr);
      if (sup.empty()) {
        pl->bw_after[g] = bandwidth_of(gr.n_edges, gr.src, gr.dst, where.data());
      } else {
        int64_t bw = 0;
        for (int64_t e = 0; e < gr.n_edges; ++e)
          if (!is_sup[gr.src[e]] && !is_sup[gr.dst[e]]) {
            const int64_t a = where[gr.src[e]], b = where[gr.dst[e]];
            bw = std::max(bw, a > b ? a - b : b - a);
          }
        pl->bw_after[g] = bw;
      }
    }
  };
  unsigned nt = std::max(1u, std::min(std::thread::hardware_concurrency(), 16u));
  nt = std::min<unsigned>(nt, (unsigned)n_graphs);
  std::vector<std::thread> pool;
  for (unsigned t = 1; t < nt; ++t) pool.emplace_back(worker);
  worker();
  for (auto& t : pool) t.join();

  // gather table and segments
  pl->gather.resize(pl->n_real);
  for (int32_t g = 0; g < pl->n_packed; ++g) {
    const bg_graph& gr = graphs[g];
    const int32_t* pg = pl->perm.data() + pl->node_base[g];
    const int32_t o = pl->offset[g];
    for (int32_t i = 0; i < gr.n_nodes; ++i) pl->gather[o + i] = (int32_t)(pl->node_base[g] + pg[i]);
    pl->seg_off.push_back(o);
    pl->seg_cnt.push_back(gr.n_nodes);
    pl->bw_before_max = std::max(pl->bw_before_max, pl->bw_before[g]);
    pl->bw_after_max = std::max(pl->bw_after_max, pl->bw_after[g]);
    pl->n_edges_in += gr.n_edges;
    pl->n_super += pl->nsup[g];
  }

  // Deduplicated edges in supergraph positions and their bits, graph by graph on the host
  // threads.  Packed graphs share no node, so each graph's sorted unique keys are a contiguous
  // run of the global sorted order, and every mask word a graph sets (forward: a row of one of its
  // targets; transposed: a row of one of its sources) belongs to that graph alone.
  const size_t tile_words = (size_t)S * pl->W32;
  const size_t nwords = (size_t)pl->K * 3 * P * tile_words;
  pl->masks.assign(nwords, 0u);
  pl->masksT.assign(nwords, 0u);
  std::vector<int64_t> uniq(pl->n_packed, 0), kept(pl->n_packed, 0), dropped(pl->n_packed, 0);
  std::vector<std::vector<int32_t>> sup_e(pl->n_packed);
  std::atomic<int32_t> next_g{0};
  auto edge_worker = [&]() {
    std::vector<uint64_t> keys;
    std::vector<int32_t> where;
    for (;;) {
      const int32_t g = next_g.fetch_add(1);
      if (g >= pl->n_packed) return;
      const bg_graph& gr = graphs[g];
      const int32_t* pg = pl->perm.data() + pl->node_base[g];
      const int32_t o = pl->offset[g];
      where.resize(gr.n_nodes);
      for (int32_t i = 0; i < gr.n_nodes; ++i) where[pg[i]] = i;
      keys.clear();
      for (int64_t e = 0; e < gr.n_edges; ++e) {
        const uint64_t tgt = (uint64_t)(o + where[gr.dst[e]]);
        const uint64_t srcp = (uint64_t)(o + where[gr.src[e]]);
        // target (28 bits) | source (28 bits) | type (6 bits) -> unique key, sorted by target
        keys.push_back((tgt << 34) | (srcp << 6) | (uint64_t)gr.etype[e]);
      }
      std::sort(keys.begin(), keys.end());
      keys.erase(std::unique(keys.begin(), keys.end()), keys.end());
      uniq[g] = (int64_t)keys.size();
      const int64_t sup_end = o + pl->nsup[g];  // the graph's supernodes: positions [o, sup_end)
      for (uint64_t key : keys) {
        const int64_t i = (int64_t)(key >> 34);
        const int64_t j = (int64_t)((key >> 6) & ((1ull << 28) - 1));
        const int32_t p = (int32_t)(key & 63);
        if (i < sup_end || j < sup_end) {
          // a supernode end: kept, propagated by the supernode rows and columns
          ++kept[g];
          sup_e[g].insert(sup_e[g].end(), {(int32_t)i, (int32_t)j, p});
          continue;
        }
        const int64_t bi = i / S, bj = j / S;
        if (bj - bi < -1 || bj - bi > 1) { ++dropped[g]; continue; }
        ++kept[g];
        const int64_t ri = i % S, cj = j % S;
        // forward: block-row bi, diagonal slot (bj - bi + 1), row ri, bit cj
        const size_t f = ((((size_t)bi * 3 + (size_t)(bj - bi + 1)) * P + p) * S + ri) * pl->W32 + cj / 32;
        pl->masks[f] |= 1u << (cj % 32);
        // transposed: source block bj, target slot (bi - bj + 1), row cj, bit ri
        const size_t t = ((((size_t)bj * 3 + (size_t)(bi - bj + 1)) * P + p) * S + cj) * pl->W32 + ri / 32;
        pl->masksT[t] |= 1u << (ri % 32);
      }
    }
  };
  unsigned ne = std::max(1u, std::min(std::thread::hardware_concurrency(), 16u));
  ne = std::min<unsigned>(ne, (unsigned)pl->n_packed);
  std::vector<std::thread> epool;
  for (unsigned t = 1; t < ne; ++t) epool.emplace_back(edge_worker);
  edge_worker();
  for (auto& t : epool) t.join();
  for (int32_t g = 0; g < pl->n_packed; ++g) {
    pl->n_unique += uniq[g];
    pl->n_kept += kept[g];
    pl->n_dropped += dropped[g];
    // graphs occupy ascending position ranges, so the concatenation stays sorted
    pl->sup_edges.insert(pl->sup_edges.end(), sup_e[g].begin(), sup_e[g].end());
  }
  *out = pl;
  return BG_OK;
}

// Block-row partition of a plan (Eq. 3: block-row k couples only to block-rows k - 1 and k + 1).
// Part `part` of n_parts owns a contiguous range of whole units of max(128, S) rows (a 128-row
// tile of 128 / S block-rows when S <= 128, one block-row otherwise); its local plan spans that
// range plus one unit of halo on each side (clipped at the ends).  The forward tiles keep only the rows the part owns as targets and the
// transposed tiles only the rows it owns as sources, so with the halo rows of E (forward) or dY
// (backward) copied in from the neighbours the part's own rows of Y and dE are exact, the halo
// rows of Y and dE come out 0, and its dW, db are the sums over its own source rows: summed over
// the parts they give the whole plan's.
int bg_plan_partition_build(const bg_plan* full, int32_t n_parts, int32_t part, bg_plan** out,
                            bg_part_info* info) {
  if (!full || !out || !info) return bg_fail(BG_EINVAL, "NULL argument");
  *out = nullptr;
  if (full->n_super > 0) return bg_fail(BG_EINVAL, "plans with supernodes cannot be partitioned");
  const int32_t S = full->S, K = full->K, P = full->P;
  const int32_t unit = S >= 128 ? 1 : 128 / S;  // block-rows per unit
  const int32_t n_units = (K + unit - 1) / unit;
  if (n_parts < 1 || n_parts > n_units) return bg_fail(BG_EINVAL, "n_parts must be in [1, units of max(128, S) rows]");
  if (part < 0 || part >= n_parts) return bg_fail(BG_EINVAL, "part out of range");
  const int32_t u0 = (int32_t)((int64_t)n_units * part / n_parts);
  const int32_t u1 = (int32_t)((int64_t)n_units * (part + 1) / n_parts);
  const int32_t k0 = u0 * unit, k1 = std::min(K, u1 * unit);  // own block-rows [k0, k1)
  const int32_t kb0 = std::max(0, k0 - unit), kb1 = std::min(K, k1 + unit);  // with the halo
  bg_plan* pl = new (std::nothrow) bg_plan();
  if (!pl) return bg_fail(BG_ENOMEM, "host allocation failed");
  pl->S = S; pl->P = P; pl->W32 = full->W32; pl->K = kb1 - kb0;
  pl->n_graphs = 0; pl->n_packed = 0;
  const int64_t row0 = (int64_t)kb0 * S;
  pl->n_real = (int32_t)std::max<int64_t>(0, std::min<int64_t>((int64_t)pl->K * S, full->n_real - row0));
  const size_t tile_words = (size_t)3 * P * S * full->W32;  // one block-row of tiles
  pl->masks.assign((size_t)pl->K * tile_words, 0u);
  pl->masksT.assign((size_t)pl->K * tile_words, 0u);
  for (int32_t k = k0; k < k1; ++k) {
    const size_t src = (size_t)k * tile_words, dst = (size_t)(k - kb0) * tile_words;
    std::memcpy(pl->masks.data() + dst, full->masks.data() + src, tile_words * 4);
    std::memcpy(pl->masksT.data() + dst, full->masksT.data() + src, tile_words * 4);
  }
  for (uint32_t w : pl->masks) pl->n_kept += __builtin_popcount(w);
  pl->n_unique = pl->n_kept;
  info->row0 = (int32_t)row0;
  info->n_local = pl->K * S;
  info->own_begin = (k0 - kb0) * S;
  info->own_end = (k1 - kb0) * S;
  info->halo_lo = (k0 - kb0) * S;
  info->halo_hi = (kb1 - k1) * S;
  *out = pl;
  return BG_OK;
}

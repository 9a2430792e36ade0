// CPU ORACLE -- TEST INFRASTRUCTURE ONLY.
//
// A plain, slow, fp64 implementation of what the band-GGNN hot path computes, written from the
// paper ("Fast Training of Sparse Graph Neural Networks on Dense Hardware", arXiv 1906.11786) and
// sharing no code, header, table or helper with the CUDA library.  Only the test suite, the smoke
// check and the benchmark's CPU-baseline leg may load it.  The product path never calls it.
//
// Because the band method is lossless on the edges it keeps (Section 3.2, Eq. 3 and the
// coverage rule after it), the oracle does NOT follow Algorithm 1: it computes the plain
// definition -- sparse message passing by scatter-add over the list of kept edges (Eq. 1 with
// per-type weights, Section 2) -- plus the bandwidth definition, Reverse Cuthill-McKee, sparse
// batching into a supergraph, a naive GRU cell, hand-derived backward passes, a mean-pool
// readout with squared loss, and Adam.  Each function names the passage it follows.
//
// Readings of points the paper leaves open (numbered as in the design notes):
//   c4 GRU gate convention: r, z, n rows in that order; n = tanh(Wi_n x + b_in + r*(Wh_n h + b_hn));
//      h' = (1-z)*n + z*h; input x = summed messages, hidden h = node state.
//   c5 per-edge-type bias: each message along a type-p edge is E[u] W_p + b_p.
//   c6 adjacency is 0/1: duplicate (src, dst, type) edges count once; self-loops are allowed.
//   c7 direction: edge u->v sends u's message to v (a_vu = 1).
//   c8 RCM: symmetrised, deduplicated neighbour sets; start of each component by the George-Liu
//      pseudo-peripheral search from the unvisited node of least (degree, id); Cuthill-McKee
//      breadth-first order visiting neighbours by ascending (degree, id); components in discovery
//      order; the whole list reversed.  Keep-if-better falls back to the input order when RCM
//      does not reduce the bandwidth.
//   c9 packing: graphs in input order, contiguous, stop at the first graph that does not fit.
//   c10 an edge is kept iff its target and source block indices differ by at most one.
//   c11 padding rows of the supergraph carry state 0 through the GRU.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <utility>
#include <vector>

namespace {

typedef std::vector<std::vector<int32_t>> NbrLists;

// Symmetric, deduplicated neighbour lists without self-loops, sorted by id (reading c8).
NbrLists symmetric_neighbours(int32_t n, int64_t m, const int32_t* src, const int32_t* dst) {
  NbrLists nb(n);
  for (int64_t e = 0; e < m; ++e) {
    int32_t u = src[e], v = dst[e];
    if (u == v) continue;
    nb[u].push_back(v);
    nb[v].push_back(u);
  }
  for (auto& l : nb) {
    std::sort(l.begin(), l.end());
    l.erase(std::unique(l.begin(), l.end()), l.end());
  }
  return nb;
}

// Breadth-first level structure rooted at r (only the component of r is reached).
std::vector<std::vector<int32_t>> level_structure(int32_t r, const NbrLists& nb) {
  std::vector<char> seen(nb.size(), 0);
  std::vector<std::vector<int32_t>> levels;
  std::vector<int32_t> cur{r};
  seen[r] = 1;
  while (!cur.empty()) {
    levels.push_back(cur);
    std::vector<int32_t> next;
    for (int32_t u : cur)
      for (int32_t v : nb[u])
        if (!seen[v]) { seen[v] = 1; next.push_back(v); }
    cur.swap(next);
  }
  return levels;
}

bool less_deg_id(const NbrLists& nb, int32_t a, int32_t b) {
  size_t da = nb[a].size(), db = nb[b].size();
  return da != db ? da < db : a < b;
}

}  // namespace

extern "C" {

// Bandwidth (Section 2, "Sparse numerical linear algebra"): the smallest B >= 0 such that
// a_ij = 0 whenever |i - j| > B.  pos[v] is node v's position (NULL = identity); edges of all
// types count.
int64_t orc_bandwidth(int32_t n, int64_t m, const int32_t* src, const int32_t* dst,
                      const int32_t* pos) {
  (void)n;
  int64_t bw = 0;
  for (int64_t e = 0; e < m; ++e) {
    int64_t i = pos ? pos[dst[e]] : dst[e];
    int64_t j = pos ? pos[src[e]] : src[e];
    int64_t d = i > j ? i - j : j - i;
    if (d > bw) bw = d;
  }
  return bw;
}

// Reverse Cuthill-McKee ordering (Section 2 and Section 3.1; tie-breaking per reading c8).
// Writes perm[new_position] = old_id.  Returns 0, or -1 on invalid input.
int orc_rcm(int32_t n, int64_t m, const int32_t* src, const int32_t* dst, int keep_if_better,
            int32_t* perm) {
  if (n < 0 || m < 0) return -1;
  for (int64_t e = 0; e < m; ++e)
    if (src[e] < 0 || src[e] >= n || dst[e] < 0 || dst[e] >= n) return -1;
  NbrLists nb = symmetric_neighbours(n, m, src, dst);
  std::vector<char> placed(n, 0);
  std::vector<int32_t> order;
  order.reserve(n);
  while ((int32_t)order.size() < n) {
    // least (degree, id) among nodes not yet placed
    int32_t r = -1;
    for (int32_t v = 0; v < n; ++v)
      if (!placed[v] && (r < 0 || less_deg_id(nb, v, r))) r = v;
    // George-Liu pseudo-peripheral node: move to the least (degree, id) node of the last level
    // while that strictly increases the eccentricity.
    auto levels = level_structure(r, nb);
    for (;;) {
      const auto& last = levels.back();
      int32_t x = last[0];
      for (int32_t v : last)
        if (less_deg_id(nb, v, x)) x = v;
      auto lx = level_structure(x, nb);
      if (lx.size() > levels.size()) {
        r = x;
        levels.swap(lx);
      } else {
        break;
      }
    }
    // Cuthill-McKee breadth-first numbering from r.
    std::vector<int32_t> queue{r};
    placed[r] = 1;
    for (size_t head = 0; head < queue.size(); ++head) {
      int32_t u = queue[head];
      order.push_back(u);
      std::vector<int32_t> fresh;
      for (int32_t v : nb[u])
        if (!placed[v]) fresh.push_back(v);
      std::sort(fresh.begin(), fresh.end(),
                [&](int32_t a, int32_t b) { return less_deg_id(nb, a, b); });
      for (int32_t v : fresh) { placed[v] = 1; queue.push_back(v); }
    }
  }
  std::reverse(order.begin(), order.end());
  if (keep_if_better) {
    std::vector<int32_t> pos(n);
    for (int32_t i = 0; i < n; ++i) pos[order[i]] = i;
    if (orc_bandwidth(n, m, src, dst, pos.data()) > orc_bandwidth(n, m, src, dst, nullptr))
      for (int32_t i = 0; i < n; ++i) order[i] = i;
  }
  std::memcpy(perm, order.data(), sizeof(int32_t) * n);
  return 0;
}

// Reachability preprocessing (Section 4 "Reachability preprocessing"): with T propagation steps
// only nodes from which some candidate node is reachable along at most T edges affect the
// candidates' final states, so the others are discarded.  Written as the definition: R_0 = the
// candidates; R_k = R_{k-1} plus every source u of an edge u -> v with v in R_{k-1}; keep R_T.
// keep[v] = 1 for kept nodes.  Returns the number kept, or -1 on invalid input.
int32_t orc_reach(int32_t n, int64_t m, const int32_t* src, const int32_t* dst,
                  const int32_t* cand, int32_t n_cand, int32_t T, uint8_t* keep) {
  if (n < 0 || m < 0 || n_cand < 0 || T < 0) return -1;
  for (int64_t e = 0; e < m; ++e)
    if (src[e] < 0 || src[e] >= n || dst[e] < 0 || dst[e] >= n) return -1;
  std::vector<uint8_t> in(n, 0);
  for (int32_t i = 0; i < n_cand; ++i) {
    if (cand[i] < 0 || cand[i] >= n) return -1;
    in[cand[i]] = 1;
  }
  for (int32_t k = 1; k <= T; ++k) {
    std::vector<uint8_t> next(in);
    for (int64_t e = 0; e < m; ++e)
      if (in[dst[e]]) next[src[e]] = 1;
    in.swap(next);
  }
  int32_t kept = 0;
  for (int32_t v = 0; v < n; ++v) {
    keep[v] = in[v];
    kept += in[v];
  }
  return kept;
}

// Number of blocks K the supergraph gets: capacity_blocks, or ceil(sum n / S) when 0, and at
// least one (reading c9: a batch with no nodes is one block of padding).
int32_t orc_num_blocks(int32_t n_graphs, const int32_t* n_nodes, int32_t S, int32_t capacity_blocks) {
  if (capacity_blocks > 0) return capacity_blocks;
  int64_t tot = 0;
  for (int32_t g = 0; g < n_graphs; ++g) tot += n_nodes[g];
  const int64_t k = (tot + S - 1) / S;
  return (int32_t)(k > 0 ? k : 1);
}

// Sparse batching into one supergraph (Section 2 "Sparse batching", Section 3.1) and the
// block-tridiagonal cover of Eq. 3.
//
// Graph g's edges are src/dst/etype[edge_off[g] .. edge_off[g+1]) with graph-local ids.
// flags bit 0: reorder each graph by RCM; bit 1: keep-if-better; bit 2: supernodes.
// Supernodes (the "supernode" propagation primitive of Section 6: some nodes may exchange
// messages with every node, through the first rows and columns of the adjacency): a node with at
// least super_min_degree distinct neighbours (edges of any type and direction, self-loops not
// counted) is a supernode, at most max_super per graph, highest degree first (ties: lower id).  A
// graph's supernodes take its first positions in that order, the RCM order of the graph without
// them follows, and every edge with a supernode end is kept whatever its block distance; the
// band masks hold the other kept edges only.  bw_after then measures the edges without a
// supernode end.
// Outputs (caller-owned):
//   perm[node_off[g] + new] = old          (node_off = prefix sums of n_nodes; every graph)
//   offset[g] = first supergraph position of g, or -1 if it was not packed
//   info[0..7] = K, n_packed, n_real, n_unique_edges, n_kept, n_dropped, bw_before_max, bw_after_max
//   masks: bit (k, d+1, p, r, c) of byte ((((k*3 + d+1)*P + p)*S + r)*(S/8) + c/8), bit c%8, is 1
//          iff the supergraph has a type-p band edge from position (k+d)*S + c to position
//          k*S + r; masks may be NULL.
//   kept_dst/kept_src/kept_type (capacity = total edges): the kept, deduplicated edges in
//          supergraph positions, sorted by (dst, src, type); may be NULL.  kept_super (may be
//          NULL) marks those with a supernode end.
//   is_super (K*S bytes, may be NULL): 1 at the positions of supernodes.
//   bw_before/bw_after per graph (may be NULL).
// Returns 0, or -1 on invalid input.
int orc_layout(int32_t n_graphs, const int32_t* n_nodes, const int64_t* edge_off,
               const int32_t* src, const int32_t* dst, const int32_t* etype, int32_t P, int32_t S,
               int32_t capacity_blocks, int32_t flags, int32_t* perm, int32_t* offset,
               int64_t* info, uint8_t* masks, int32_t* kept_dst, int32_t* kept_src,
               int32_t* kept_type, int64_t* bw_before, int64_t* bw_after,
               int32_t super_min_degree, int32_t max_super, uint8_t* kept_super,
               uint8_t* is_super) {
  if (n_graphs < 0 || P < 1 || S < 8 || S % 8 != 0) return -1;
  int32_t K = orc_num_blocks(n_graphs, n_nodes, S, capacity_blocks);
  int64_t cap = (int64_t)K * S;
  int64_t node_off = 0, next_pos = 0;
  bool stopped = false;
  int32_t n_packed = 0;
  int64_t bwb_max = 0, bwa_max = 0;
  std::vector<std::pair<std::pair<int64_t, int64_t>, int32_t>> edges;  // ((dst, src), type)
  std::vector<uint8_t> sup_at((size_t)cap, 0);
  for (int32_t g = 0; g < n_graphs; ++g) {
    int32_t n = n_nodes[g];
    int64_t e0 = edge_off[g], e1 = edge_off[g + 1];
    if (n < 0 || e1 < e0) return -1;
    for (int64_t e = e0; e < e1; ++e)
      if (src[e] < 0 || src[e] >= n || dst[e] < 0 || dst[e] >= n || etype[e] < 0 ||
          etype[e] >= P)
        return -1;
    // supernodes first (bit 2), then the rest in RCM (bit 0) or input order
    std::vector<int32_t> sup;
    if (flags & 4) {
      NbrLists nb = symmetric_neighbours(n, e1 - e0, src + e0, dst + e0);
      for (int32_t v = 0; v < n; ++v)
        if ((int64_t)nb[v].size() >= super_min_degree) sup.push_back(v);
      std::sort(sup.begin(), sup.end(), [&](int32_t a, int32_t b) {
        return nb[a].size() != nb[b].size() ? nb[a].size() > nb[b].size() : a < b;
      });
      if ((int32_t)sup.size() > max_super) sup.resize(std::max(0, max_super));
    }
    std::vector<char> sflag(n, 0);
    for (int32_t v : sup) sflag[v] = 1;
    std::vector<int32_t> rest, rid(n, -1);
    for (int32_t v = 0; v < n; ++v)
      if (!sflag[v]) { rid[v] = (int32_t)rest.size(); rest.push_back(v); }
    std::vector<int32_t> rs, rd;
    for (int64_t e = e0; e < e1; ++e)
      if (!sflag[src[e]] && !sflag[dst[e]]) { rs.push_back(rid[src[e]]); rd.push_back(rid[dst[e]]); }
    const int32_t nr = (int32_t)rest.size();
    std::vector<int32_t> pr(nr);
    if (flags & 1) {
      if (orc_rcm(nr, (int64_t)rs.size(), rs.data(), rd.data(), (flags & 2) ? 1 : 0, pr.data()))
        return -1;
    } else {
      for (int32_t i = 0; i < nr; ++i) pr[i] = i;
    }
    std::vector<int32_t> p(sup);
    for (int32_t i = 0; i < nr; ++i) p.push_back(rest[pr[i]]);
    std::memcpy(perm + node_off, p.data(), sizeof(int32_t) * n);
    std::vector<int32_t> pos(n);
    for (int32_t i = 0; i < n; ++i) pos[p[i]] = i;
    int64_t bwb = orc_bandwidth(n, e1 - e0, src + e0, dst + e0, nullptr);
    int64_t bwa = 0;
    for (int64_t e = e0; e < e1; ++e)
      if (!sflag[src[e]] && !sflag[dst[e]])
        bwa = std::max<int64_t>(bwa, std::abs((int64_t)pos[dst[e]] - (int64_t)pos[src[e]]));
    if (bw_before) bw_before[g] = bwb;
    if (bw_after) bw_after[g] = bwa;
    if (!stopped && next_pos + n <= cap) {
      offset[g] = (int32_t)next_pos;
      ++n_packed;
      bwb_max = std::max(bwb_max, bwb);
      bwa_max = std::max(bwa_max, bwa);
      for (size_t i = 0; i < sup.size(); ++i) sup_at[(size_t)next_pos + i] = 1;
      for (int64_t e = e0; e < e1; ++e)
        edges.push_back({{next_pos + pos[dst[e]], next_pos + pos[src[e]]}, etype[e]});
      next_pos += n;
    } else {
      stopped = true;
      offset[g] = -1;
    }
    node_off += n;
  }
  std::sort(edges.begin(), edges.end());
  edges.erase(std::unique(edges.begin(), edges.end()), edges.end());
  if (masks) std::memset(masks, 0, (size_t)K * 3 * P * S * (S / 8));
  if (is_super) std::memcpy(is_super, sup_at.data(), (size_t)cap);
  int64_t kept = 0, dropped = 0;
  for (const auto& ed : edges) {
    int64_t i = ed.first.first, j = ed.first.second;
    int32_t t = ed.second;
    int64_t k = i / S, c = j / S, d = c - k;
    const bool via_super = sup_at[(size_t)i] || sup_at[(size_t)j];
    if (!via_super && (d < -1 || d > 1)) { ++dropped; continue; }
    if (masks && !via_super) {
      int64_t r = i % S, cc = j % S;
      size_t byte = ((((size_t)k * 3 + (size_t)(d + 1)) * P + t) * S + r) * (S / 8) + cc / 8;
      masks[byte] |= (uint8_t)(1u << (cc % 8));
    }
    if (kept_dst) {
      kept_dst[kept] = (int32_t)i;
      kept_src[kept] = (int32_t)j;
      kept_type[kept] = t;
    }
    if (kept_super) kept_super[kept] = via_super ? 1 : 0;
    ++kept;
  }
  info[0] = K; info[1] = n_packed; info[2] = next_pos; info[3] = (int64_t)edges.size();
  info[4] = kept; info[5] = dropped; info[6] = bwb_max; info[7] = bwa_max;
  return 0;
}

// Multi-type message passing on the kept edges (Eq. 1 with separate W_p per type, Section 2;
// per-type bias, Appendix D; messages summed, not averaged, Appendix D):
//   Y[v] = sum over kept edges (u -> v, type p) of ( E[u] W_p + b_p ).
// E [N][H], W [P][H][H] with W[p][h_in][h_out], b [P][H] or NULL, Y [N][H] (overwritten).
void orc_propagate_fwd(int32_t N, int32_t P, int32_t H, int64_t n_edges, const int32_t* e_dst,
                       const int32_t* e_src, const int32_t* e_type, const double* E,
                       const double* W, const double* b, double* Y) {
  // messages M[p][u][:] = E[u] W_p + b_p for every node and type (triple loop)
  std::vector<double> M((size_t)P * N * H);
  for (int32_t p = 0; p < P; ++p)
    for (int32_t u = 0; u < N; ++u)
      for (int32_t ho = 0; ho < H; ++ho) {
        double s = b ? b[(size_t)p * H + ho] : 0.0;
        for (int32_t hi = 0; hi < H; ++hi)
          s += E[(size_t)u * H + hi] * W[((size_t)p * H + hi) * H + ho];
        M[((size_t)p * N + u) * H + ho] = s;
      }
  std::memset(Y, 0, sizeof(double) * (size_t)N * H);
  for (int64_t e = 0; e < n_edges; ++e) {
    const double* m = &M[((size_t)e_type[e] * N + e_src[e]) * H];
    double* y = &Y[(size_t)e_dst[e] * H];
    for (int32_t h = 0; h < H; ++h) y[h] += m[h];
  }
}

// Backward of orc_propagate_fwd, derived by hand from it:
//   dM_p[u] = sum over kept edges (u -> v, type p) of dY[v]
//   dE[u]   = sum_p dM_p[u] W_p^T,   dW_p = sum_u E[u]^T dM_p[u],   db_p = sum_u dM_p[u].
// Outputs are overwritten; db may be NULL.
void orc_propagate_bwd(int32_t N, int32_t P, int32_t H, int64_t n_edges, const int32_t* e_dst,
                       const int32_t* e_src, const int32_t* e_type, const double* E,
                       const double* W, const double* dY, double* dE, double* dW, double* db) {
  std::vector<double> dM((size_t)P * N * H, 0.0);
  for (int64_t e = 0; e < n_edges; ++e) {
    double* g = &dM[((size_t)e_type[e] * N + e_src[e]) * H];
    const double* y = &dY[(size_t)e_dst[e] * H];
    for (int32_t h = 0; h < H; ++h) g[h] += y[h];
  }
  std::memset(dE, 0, sizeof(double) * (size_t)N * H);
  std::memset(dW, 0, sizeof(double) * (size_t)P * H * H);
  if (db) std::memset(db, 0, sizeof(double) * (size_t)P * H);
  for (int32_t p = 0; p < P; ++p)
    for (int32_t u = 0; u < N; ++u) {
      const double* g = &dM[((size_t)p * N + u) * H];
      for (int32_t hi = 0; hi < H; ++hi) {
        double s = 0.0;
        for (int32_t ho = 0; ho < H; ++ho) s += g[ho] * W[((size_t)p * H + hi) * H + ho];
        dE[(size_t)u * H + hi] += s;
        for (int32_t ho = 0; ho < H; ++ho)
          dW[((size_t)p * H + hi) * H + ho] += E[(size_t)u * H + hi] * g[ho];
      }
      if (db)
        for (int32_t ho = 0; ho < H; ++ho) db[(size_t)p * H + ho] += g[ho];
    }
}

static double sigmoid(double x) { return 1.0 / (1.0 + std::exp(-x)); }

// GRU cell (Cho et al., named in Section 2 and Algorithm 1; gate convention per reading c4):
// X = messages [N][H], Hs = states [N][H], W_ih/W_hh [3H][H] (rows r, z, n), b_ih/b_hh [3H].
// Rows >= n_real are padding and get state 0 (reading c11).  Hn [N][H] is overwritten.
void orc_gru_fwd(int32_t N, int32_t H, int32_t n_real, const double* X, const double* Hs,
                 const double* W_ih, const double* W_hh, const double* b_ih, const double* b_hh,
                 double* Hn) {
  std::vector<double> gi(3 * H), gh(3 * H);
  for (int32_t i = 0; i < N; ++i) {
    if (i >= n_real) {
      for (int32_t h = 0; h < H; ++h) Hn[(size_t)i * H + h] = 0.0;
      continue;
    }
    for (int32_t o = 0; o < 3 * H; ++o) {
      double a = b_ih[o], c = b_hh[o];
      for (int32_t h = 0; h < H; ++h) {
        a += W_ih[(size_t)o * H + h] * X[(size_t)i * H + h];
        c += W_hh[(size_t)o * H + h] * Hs[(size_t)i * H + h];
      }
      gi[o] = a; gh[o] = c;
    }
    for (int32_t h = 0; h < H; ++h) {
      double r = sigmoid(gi[h] + gh[h]);
      double z = sigmoid(gi[H + h] + gh[H + h]);
      double nn = std::tanh(gi[2 * H + h] + r * gh[2 * H + h]);
      Hn[(size_t)i * H + h] = (1.0 - z) * nn + z * Hs[(size_t)i * H + h];
    }
  }
}

// Backward of orc_gru_fwd, derived by hand.  Given dHn, writes dX and dHs (overwritten) and
// ADDS into dW_ih, dW_hh, db_ih, db_hh.
void orc_gru_bwd(int32_t N, int32_t H, int32_t n_real, const double* X, const double* Hs,
                 const double* W_ih, const double* W_hh, const double* b_ih, const double* b_hh,
                 const double* dHn, double* dX, double* dHs, double* dW_ih, double* dW_hh,
                 double* db_ih, double* db_hh) {
  std::vector<double> gi(3 * H), gh(3 * H), dgi(3 * H), dgh(3 * H);
  for (int32_t i = 0; i < N; ++i) {
    double* dx = &dX[(size_t)i * H];
    double* dh = &dHs[(size_t)i * H];
    if (i >= n_real) {
      for (int32_t h = 0; h < H; ++h) { dx[h] = 0.0; dh[h] = 0.0; }
      continue;
    }
    const double* x = &X[(size_t)i * H];
    const double* hs = &Hs[(size_t)i * H];
    for (int32_t o = 0; o < 3 * H; ++o) {
      double a = b_ih[o], c = b_hh[o];
      for (int32_t h = 0; h < H; ++h) {
        a += W_ih[(size_t)o * H + h] * x[h];
        c += W_hh[(size_t)o * H + h] * hs[h];
      }
      gi[o] = a; gh[o] = c;
    }
    for (int32_t h = 0; h < H; ++h) {
      double r = sigmoid(gi[h] + gh[h]);
      double z = sigmoid(gi[H + h] + gh[H + h]);
      double nn = std::tanh(gi[2 * H + h] + r * gh[2 * H + h]);
      double g = dHn[(size_t)i * H + h];
      double dn = g * (1.0 - z);
      double dz = g * (hs[h] - nn);
      double dan = dn * (1.0 - nn * nn);
      double dr = dan * gh[2 * H + h];
      double daz = dz * z * (1.0 - z);
      double dar = dr * r * (1.0 - r);
      dgi[h] = dar; dgi[H + h] = daz; dgi[2 * H + h] = dan;
      dgh[h] = dar; dgh[H + h] = daz; dgh[2 * H + h] = dan * r;
      dh[h] = g * z;
    }
    for (int32_t h = 0; h < H; ++h) dx[h] = 0.0;
    for (int32_t o = 0; o < 3 * H; ++o) {
      db_ih[o] += dgi[o];
      db_hh[o] += dgh[o];
      for (int32_t h = 0; h < H; ++h) {
        dx[h] += W_ih[(size_t)o * H + h] * dgi[o];
        dh[h] += W_hh[(size_t)o * H + h] * dgh[o];
        dW_ih[(size_t)o * H + h] += dgi[o] * x[h];
        dW_hh[(size_t)o * H + h] += dgh[o] * hs[h];
      }
    }
  }
}

// T GGNN steps, Eq. 1 with P edge types: E(t+1) = GRU(sum_p A_p (E(t) W_p + b_p), E(t)).
// Es [(T+1)][N][H] receives E(0..T) (Es[0] must hold E(0) on entry); Ys [T][N][H] the messages.
void orc_ggnn_fwd(int32_t N, int32_t P, int32_t H, int32_t T, int32_t n_real, int64_t n_edges,
                  const int32_t* e_dst, const int32_t* e_src, const int32_t* e_type,
                  const double* W, const double* b, const double* W_ih, const double* W_hh,
                  const double* b_ih, const double* b_hh, double* Es, double* Ys) {
  size_t NH = (size_t)N * H;
  for (int32_t t = 0; t < T; ++t) {
    orc_propagate_fwd(N, P, H, n_edges, e_dst, e_src, e_type, Es + t * NH, W, b, Ys + t * NH);
    orc_gru_fwd(N, H, n_real, Ys + t * NH, Es + t * NH, W_ih, W_hh, b_ih, b_hh,
                Es + (t + 1) * NH);
  }
}

// Backward through orc_ggnn_fwd (reverse over t).  dET is the gradient at E(T); writes dE0 and
// overwrites all parameter gradients.
void orc_ggnn_bwd(int32_t N, int32_t P, int32_t H, int32_t T, int32_t n_real, int64_t n_edges,
                  const int32_t* e_dst, const int32_t* e_src, const int32_t* e_type,
                  const double* W, const double* b, const double* W_ih, const double* W_hh,
                  const double* b_ih, const double* b_hh, const double* Es, const double* Ys,
                  const double* dET, double* dE0, double* dW, double* db, double* dW_ih,
                  double* dW_hh, double* db_ih, double* db_hh) {
  (void)b;
  size_t NH = (size_t)N * H;
  std::vector<double> g(dET, dET + NH), dX(NH), dHs(NH), dEp(NH);
  std::vector<double> dWt((size_t)P * H * H), dbt((size_t)P * H);
  std::memset(dW, 0, sizeof(double) * P * H * H);
  std::memset(db, 0, sizeof(double) * P * H);
  std::memset(dW_ih, 0, sizeof(double) * 3 * H * H);
  std::memset(dW_hh, 0, sizeof(double) * 3 * H * H);
  std::memset(db_ih, 0, sizeof(double) * 3 * H);
  std::memset(db_hh, 0, sizeof(double) * 3 * H);
  for (int32_t t = T - 1; t >= 0; --t) {
    orc_gru_bwd(N, H, n_real, Ys + t * NH, Es + t * NH, W_ih, W_hh, b_ih, b_hh, g.data(),
                dX.data(), dHs.data(), dW_ih, dW_hh, db_ih, db_hh);
    orc_propagate_bwd(N, P, H, n_edges, e_dst, e_src, e_type, Es + t * NH, W, dX.data(),
                      dEp.data(), dWt.data(), dbt.data());
    for (size_t i = 0; i < NH; ++i) g[i] = dHs[i] + dEp[i];
    for (size_t i = 0; i < dWt.size(); ++i) dW[i] += dWt[i];
    for (size_t i = 0; i < dbt.size(); ++i) db[i] += dbt[i];
  }
  std::memcpy(dE0, g.data(), sizeof(double) * NH);
}

// Per-graph mean-pool readout with a linear output and squared loss (the training workload's
// readout; the paper's own readout, Section 2 "Variable misuse", needs candidate labels):
//   pool_g = mean of E[offset_g .. offset_g + n_g),  pred_g = w_out . pool_g,
//   loss = 1/2 sum_g (pred_g - y_g)^2.
// Writes loss, dE (overwritten; rows outside every graph get 0) and dw_out.
void orc_readout_loss(int32_t N, int32_t H, int32_t n_g, const int32_t* offset,
                      const int32_t* count, const double* E, const double* w_out,
                      const double* target, double* loss, double* dE, double* dw_out) {
  std::memset(dE, 0, sizeof(double) * (size_t)N * H);
  std::memset(dw_out, 0, sizeof(double) * H);
  double L = 0.0;
  std::vector<double> pool(H);
  for (int32_t g = 0; g < n_g; ++g) {
    for (int32_t h = 0; h < H; ++h) pool[h] = 0.0;
    for (int32_t i = offset[g]; i < offset[g] + count[g]; ++i)
      for (int32_t h = 0; h < H; ++h) pool[h] += E[(size_t)i * H + h];
    for (int32_t h = 0; h < H; ++h) pool[h] /= count[g];
    double pred = 0.0;
    for (int32_t h = 0; h < H; ++h) pred += w_out[h] * pool[h];
    double r = pred - target[g];
    L += 0.5 * r * r;
    for (int32_t h = 0; h < H; ++h) dw_out[h] += r * pool[h];
    for (int32_t i = offset[g]; i < offset[g] + count[g]; ++i)
      for (int32_t h = 0; h < H; ++h) dE[(size_t)i * H + h] = r * w_out[h] / count[g];
  }
  *loss = L;
}

// Adam (Kingma & Ba), bias-corrected, one step `t` >= 1, in place on param/m/v.
void orc_adam(int64_t n, double* param, double* m, double* v, const double* grad, double lr,
              double b1, double b2, double eps, int32_t t) {
  double c1 = 1.0 - std::pow(b1, t), c2 = 1.0 - std::pow(b2, t);
  for (int64_t i = 0; i < n; ++i) {
    m[i] = b1 * m[i] + (1.0 - b1) * grad[i];
    v[i] = b2 * v[i] + (1.0 - b2) * grad[i] * grad[i];
    param[i] -= lr * (m[i] / c1) / (std::sqrt(v[i] / c2) + eps);
  }
}

}  // extern "C"

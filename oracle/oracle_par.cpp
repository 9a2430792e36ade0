// CPU ORACLE, multi-threaded pull-based variant -- TEST INFRASTRUCTURE ONLY (CPU baseline timing).
//
// The same computation as oracle.cpp's propagation, GRU and GGNN functions, restated so that the
// host cores can share it (OpenMP): every output element is owned by one thread and gathers its
// terms ("pull") instead of scattering them, in the same order as the single-threaded oracle adds
// them.  Floating-point addition is not associative, so that order is the whole contract: each
// sum below starts from the same value and adds the same terms in the same order as its
// counterpart in oracle.cpp, and the results are equal to the last bit (a CPU test checks this).
//   - messages Y[v]: in-edges of v in edge-list order (a stable bucket sort by target);
//   - dM_p[u]: out-edges of u of type p in edge-list order (a stable bucket sort by source);
//   - dE[u]: types in ascending order; dW, db, and the GRU weight and bias gradients: nodes in
//     ascending order.
// Nothing here is used by the library; only the benchmark's CPU-baseline leg and the tests load
// it.  Shares no code with the CUDA path.
#include <cmath>
#include <cstdint>
#include <cstring>
#include <vector>

#ifdef _OPENMP
#include <omp.h>
#endif

namespace {

double sigmoid_p(double x) { return 1.0 / (1.0 + std::exp(-x)); }

// Edge ids grouped by key[e] (stable: ascending e within a group): CSR offsets and ids.
void bucket(int32_t n_keys, int64_t m, const int32_t* key, std::vector<int64_t>& off,
            std::vector<int64_t>& ids) {
  off.assign((size_t)n_keys + 1, 0);
  for (int64_t e = 0; e < m; ++e) ++off[(size_t)key[e] + 1];
  for (int32_t k = 0; k < n_keys; ++k) off[k + 1] += off[k];
  std::vector<int64_t> pos(off.begin(), off.end() - 1);
  ids.resize((size_t)m);
  for (int64_t e = 0; e < m; ++e) ids[(size_t)pos[key[e]]++] = e;
}

void set_threads(int32_t nt) {
#ifdef _OPENMP
  if (nt > 0) omp_set_num_threads(nt);
#else
  (void)nt;
#endif
}

void par_fwd(int32_t N, int32_t P, int32_t H, int64_t n_edges, const int32_t* e_dst,
             const int32_t* e_src, const int32_t* e_type, const double* E, const double* W,
             const double* b, double* Y) {
  std::vector<double> M((size_t)P * N * H);
#pragma omp parallel for schedule(static)
  for (int64_t pu = 0; pu < (int64_t)P * N; ++pu) {
    const int32_t p = (int32_t)(pu / N), u = (int32_t)(pu % N);
    for (int32_t ho = 0; ho < H; ++ho) {
      double s = b ? b[(size_t)p * H + ho] : 0.0;
      for (int32_t hi = 0; hi < H; ++hi) s += E[(size_t)u * H + hi] * W[((size_t)p * H + hi) * H + ho];
      M[((size_t)p * N + u) * H + ho] = s;
    }
  }
  std::vector<int64_t> off, ids;
  bucket(N, n_edges, e_dst, off, ids);
#pragma omp parallel for schedule(dynamic, 64)
  for (int32_t v = 0; v < N; ++v) {
    double* y = &Y[(size_t)v * H];
    for (int32_t h = 0; h < H; ++h) y[h] = 0.0;
    for (int64_t i = off[v]; i < off[v + 1]; ++i) {
      const int64_t e = ids[(size_t)i];
      const double* m = &M[((size_t)e_type[e] * N + e_src[e]) * H];
      for (int32_t h = 0; h < H; ++h) y[h] += m[h];
    }
  }
}

void par_bwd(int32_t N, int32_t P, int32_t H, int64_t n_edges, const int32_t* e_dst,
             const int32_t* e_src, const int32_t* e_type, const double* E, const double* W,
             const double* dY, double* dE, double* dW, double* db) {
  std::vector<double> dM((size_t)P * N * H, 0.0);
  std::vector<int64_t> off, ids;
  bucket(N, n_edges, e_src, off, ids);
#pragma omp parallel for schedule(dynamic, 64)
  for (int32_t u = 0; u < N; ++u)
    for (int64_t i = off[u]; i < off[u + 1]; ++i) {
      const int64_t e = ids[(size_t)i];
      double* g = &dM[((size_t)e_type[e] * N + u) * H];
      const double* y = &dY[(size_t)e_dst[e] * H];
      for (int32_t h = 0; h < H; ++h) g[h] += y[h];
    }
#pragma omp parallel for schedule(static)
  for (int32_t u = 0; u < N; ++u)
    for (int32_t hi = 0; hi < H; ++hi) {
      double acc = 0.0;
      for (int32_t p = 0; p < P; ++p) {
        const double* g = &dM[((size_t)p * N + u) * H];
        double s = 0.0;
        for (int32_t ho = 0; ho < H; ++ho) s += g[ho] * W[((size_t)p * H + hi) * H + ho];
        acc += s;
      }
      dE[(size_t)u * H + hi] = acc;
    }
#pragma omp parallel for schedule(static)
  for (int64_t ph = 0; ph < (int64_t)P * H; ++ph) {
    const int32_t p = (int32_t)(ph / H), hi = (int32_t)(ph % H);
    double* w = &dW[((size_t)p * H + hi) * H];
    for (int32_t ho = 0; ho < H; ++ho) w[ho] = 0.0;
    for (int32_t u = 0; u < N; ++u) {
      const double* g = &dM[((size_t)p * N + u) * H];
      const double e = E[(size_t)u * H + hi];
      for (int32_t ho = 0; ho < H; ++ho) w[ho] += e * g[ho];
    }
  }
  if (db) {
#pragma omp parallel for schedule(static)
    for (int32_t p = 0; p < P; ++p) {
      double* d = &db[(size_t)p * H];
      for (int32_t ho = 0; ho < H; ++ho) d[ho] = 0.0;
      for (int32_t u = 0; u < N; ++u) {
        const double* g = &dM[((size_t)p * N + u) * H];
        for (int32_t ho = 0; ho < H; ++ho) d[ho] += g[ho];
      }
    }
  }
}

void par_gru_fwd(int32_t N, int32_t H, int32_t n_real, const double* X, const double* Hs,
                 const double* W_ih, const double* W_hh, const double* b_ih, const double* b_hh,
                 double* Hn) {
#pragma omp parallel
  {
    std::vector<double> gi(3 * H), gh(3 * H);
#pragma omp for schedule(static)
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
        const double r = sigmoid_p(gi[h] + gh[h]);
        const double z = sigmoid_p(gi[H + h] + gh[H + h]);
        const double nn = std::tanh(gi[2 * H + h] + r * gh[2 * H + h]);
        Hn[(size_t)i * H + h] = (1.0 - z) * nn + z * Hs[(size_t)i * H + h];
      }
    }
  }
}

// Adds into dW_ih, dW_hh, db_ih, db_hh like oracle.cpp's orc_gru_bwd (nodes in ascending order).
void par_gru_bwd(int32_t N, int32_t H, int32_t n_real, const double* X, const double* Hs,
                 const double* W_ih, const double* W_hh, const double* b_ih, const double* b_hh,
                 const double* dHn, double* dX, double* dHs, double* dW_ih, double* dW_hh,
                 double* db_ih, double* db_hh) {
  const int32_t nr = n_real < N ? n_real : N;
  std::vector<double> DGI((size_t)nr * 3 * H), DGH((size_t)nr * 3 * H);
#pragma omp parallel
  {
    std::vector<double> gi(3 * H), gh(3 * H);
#pragma omp for schedule(static)
    for (int32_t i = 0; i < N; ++i) {
      double* dx = &dX[(size_t)i * H];
      double* dh = &dHs[(size_t)i * H];
      if (i >= n_real) {
        for (int32_t h = 0; h < H; ++h) { dx[h] = 0.0; dh[h] = 0.0; }
        continue;
      }
      const double* x = &X[(size_t)i * H];
      const double* hs = &Hs[(size_t)i * H];
      double* dgi = &DGI[(size_t)i * 3 * H];
      double* dgh = &DGH[(size_t)i * 3 * H];
      for (int32_t o = 0; o < 3 * H; ++o) {
        double a = b_ih[o], c = b_hh[o];
        for (int32_t h = 0; h < H; ++h) {
          a += W_ih[(size_t)o * H + h] * x[h];
          c += W_hh[(size_t)o * H + h] * hs[h];
        }
        gi[o] = a; gh[o] = c;
      }
      for (int32_t h = 0; h < H; ++h) {
        const double r = sigmoid_p(gi[h] + gh[h]);
        const double z = sigmoid_p(gi[H + h] + gh[H + h]);
        const double nn = std::tanh(gi[2 * H + h] + r * gh[2 * H + h]);
        const double g = dHn[(size_t)i * H + h];
        const double dn = g * (1.0 - z);
        const double dz = g * (hs[h] - nn);
        const double dan = dn * (1.0 - nn * nn);
        const double dr = dan * gh[2 * H + h];
        const double daz = dz * z * (1.0 - z);
        const double dar = dr * r * (1.0 - r);
        dgi[h] = dar; dgi[H + h] = daz; dgi[2 * H + h] = dan;
        dgh[h] = dar; dgh[H + h] = daz; dgh[2 * H + h] = dan * r;
        dh[h] = g * z;
      }
      for (int32_t h = 0; h < H; ++h) dx[h] = 0.0;
      for (int32_t o = 0; o < 3 * H; ++o)
        for (int32_t h = 0; h < H; ++h) {
          dx[h] += W_ih[(size_t)o * H + h] * dgi[o];
          dh[h] += W_hh[(size_t)o * H + h] * dgh[o];
        }
    }
#pragma omp for schedule(static)
    for (int32_t o = 0; o < 3 * H; ++o) {
      double bi = db_ih[o], bh = db_hh[o];
      for (int32_t i = 0; i < nr; ++i) {
        bi += DGI[(size_t)i * 3 * H + o];
        bh += DGH[(size_t)i * 3 * H + o];
      }
      db_ih[o] = bi; db_hh[o] = bh;
      for (int32_t h = 0; h < H; ++h) {
        double wi = dW_ih[(size_t)o * H + h], wh = dW_hh[(size_t)o * H + h];
        for (int32_t i = 0; i < nr; ++i) {
          wi += DGI[(size_t)i * 3 * H + o] * X[(size_t)i * H + h];
          wh += DGH[(size_t)i * 3 * H + o] * Hs[(size_t)i * H + h];
        }
        dW_ih[(size_t)o * H + h] = wi; dW_hh[(size_t)o * H + h] = wh;
      }
    }
  }
}

}  // namespace

extern "C" {

// Equal to the last bit to orc_propagate_fwd / orc_propagate_bwd; n_threads <= 0 keeps the
// OpenMP default (all host cores).
void orc_par_propagate_fwd(int32_t N, int32_t P, int32_t H, int64_t n_edges, const int32_t* e_dst,
                           const int32_t* e_src, const int32_t* e_type, const double* E,
                           const double* W, const double* b, double* Y, int32_t n_threads) {
  set_threads(n_threads);
  par_fwd(N, P, H, n_edges, e_dst, e_src, e_type, E, W, b, Y);
}

void orc_par_propagate_bwd(int32_t N, int32_t P, int32_t H, int64_t n_edges, const int32_t* e_dst,
                           const int32_t* e_src, const int32_t* e_type, const double* E,
                           const double* W, const double* dY, double* dE, double* dW, double* db,
                           int32_t n_threads) {
  set_threads(n_threads);
  par_bwd(N, P, H, n_edges, e_dst, e_src, e_type, E, W, dY, dE, dW, db);
}

// Equal to the last bit to orc_ggnn_fwd / orc_ggnn_bwd (same step structure).
void orc_par_ggnn_fwd(int32_t N, int32_t P, int32_t H, int32_t T, int32_t n_real, int64_t n_edges,
                      const int32_t* e_dst, const int32_t* e_src, const int32_t* e_type,
                      const double* W, const double* b, const double* W_ih, const double* W_hh,
                      const double* b_ih, const double* b_hh, double* Es, double* Ys,
                      int32_t n_threads) {
  set_threads(n_threads);
  const size_t NH = (size_t)N * H;
  for (int32_t t = 0; t < T; ++t) {
    par_fwd(N, P, H, n_edges, e_dst, e_src, e_type, Es + t * NH, W, b, Ys + t * NH);
    par_gru_fwd(N, H, n_real, Ys + t * NH, Es + t * NH, W_ih, W_hh, b_ih, b_hh, Es + (t + 1) * NH);
  }
}

void orc_par_ggnn_bwd(int32_t N, int32_t P, int32_t H, int32_t T, int32_t n_real, int64_t n_edges,
                      const int32_t* e_dst, const int32_t* e_src, const int32_t* e_type,
                      const double* W, const double* b, const double* W_ih, const double* W_hh,
                      const double* b_ih, const double* b_hh, const double* Es, const double* Ys,
                      const double* dET, double* dE0, double* dW, double* db, double* dW_ih,
                      double* dW_hh, double* db_ih, double* db_hh, int32_t n_threads) {
  (void)b;
  set_threads(n_threads);
  const size_t NH = (size_t)N * H;
  std::vector<double> g(dET, dET + NH), dX(NH), dHs(NH), dEp(NH);
  std::vector<double> dWt((size_t)P * H * H), dbt((size_t)P * H);
  std::memset(dW, 0, sizeof(double) * P * H * H);
  std::memset(db, 0, sizeof(double) * P * H);
  std::memset(dW_ih, 0, sizeof(double) * 3 * H * H);
  std::memset(dW_hh, 0, sizeof(double) * 3 * H * H);
  std::memset(db_ih, 0, sizeof(double) * 3 * H);
  std::memset(db_hh, 0, sizeof(double) * 3 * H);
  for (int32_t t = T - 1; t >= 0; --t) {
    par_gru_bwd(N, H, n_real, Ys + t * NH, Es + t * NH, W_ih, W_hh, b_ih, b_hh, g.data(),
                dX.data(), dHs.data(), dW_ih, dW_hh, db_ih, db_hh);
    par_bwd(N, P, H, n_edges, e_dst, e_src, e_type, Es + t * NH, W, dX.data(), dEp.data(),
            dWt.data(), dbt.data());
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < (int64_t)NH; ++i) g[i] = dHs[i] + dEp[i];
    for (size_t i = 0; i < dWt.size(); ++i) dW[i] += dWt[i];
    for (size_t i = 0; i < dbt.size(); ++i) db[i] += dbt[i];
  }
  std::memcpy(dE0, g.data(), sizeof(double) * NH);
}

// Threads the OpenMP runtime uses by default (1 without OpenMP).
int32_t orc_par_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

}  // extern "C"

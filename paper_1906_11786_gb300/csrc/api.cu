// C ABI of the band-GGNN library: argument checks, workspace layout, orchestration of the
// kernels, kernel timing and error reporting.  Every numeric step runs in this library's kernels.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "band_tc.h"
#include "gemm_tc.h"
#include "gru_tc.h"
#include "internal.h"
#include "kernels.h"
#include "super.h"

namespace bg {
long long launch_total();
}

// ---------------------------------------------------------------------------------- errors
static thread_local std::string t_err;

int bg_fail(int code, const std::string& msg) {
  t_err = msg;
  return code;
}
void bg_clear_error() { t_err.clear(); }

extern "C" const char* bg_last_error(void) { return t_err.c_str(); }
extern "C" int64_t bg_launch_count(void) { return (int64_t)bg::launch_total(); }

#define BG_CUDA(call)                                                                      \
  do {                                                                                     \
    cudaError_t e_ = (call);                                                               \
    if (e_ != cudaSuccess)                                                                 \
      return bg_fail(BG_ECUDA, std::string(#call) + ": " + cudaGetErrorString(e_));        \
  } while (0)

#define BG_TRY(call)          \
  do {                        \
    int rc_ = (call);         \
    if (rc_ != BG_OK) return rc_; \
  } while (0)

// ---------------------------------------------------------------------------------- profiling
namespace {
struct EvPair {
  int kid;
  cudaEvent_t a, b;
};
std::mutex g_prof_mu;
bool g_prof_on = false;
std::vector<EvPair> g_prof_events;
double g_prof_ms[BG_KID_COUNT] = {0};
int64_t g_prof_n[BG_KID_COUNT] = {0};

// Records CUDA events on `st` around a kernel while profiling is enabled.
struct KTimer {
  int kid;
  cudaStream_t st;
  cudaEvent_t a = nullptr, b = nullptr;
  KTimer(int kid_, cudaStream_t st_) : kid(kid_), st(st_) {
    std::lock_guard<std::mutex> g(g_prof_mu);
    if (!g_prof_on) return;
    if (cudaEventCreate(&a) != cudaSuccess || cudaEventCreate(&b) != cudaSuccess) {
      a = b = nullptr;
      return;
    }
    cudaEventRecord(a, st);
  }
  ~KTimer() {
    if (!a) return;
    cudaEventRecord(b, st);
    std::lock_guard<std::mutex> g(g_prof_mu);
    g_prof_events.push_back({kid, a, b});
  }
};

int status_word_ptr(int** out);
}  // namespace

namespace bg {
ProfSpan::ProfSpan(int kid, cudaStream_t st) : kid_(kid), st_(st) {
  std::lock_guard<std::mutex> g(g_prof_mu);
  if (!g_prof_on) return;
  if (cudaEventCreate(&a_) != cudaSuccess || cudaEventCreate(&b_) != cudaSuccess) {
    a_ = b_ = nullptr;
    return;
  }
  cudaEventRecord(a_, st_);
}
ProfSpan::~ProfSpan() {
  if (!a_) return;
  cudaEventRecord(b_, st_);
  std::lock_guard<std::mutex> g(g_prof_mu);
  g_prof_events.push_back({kid_, a_, b_});
}
}  // namespace bg

extern "C" int bg_profile_enable(int32_t on) {
  std::lock_guard<std::mutex> g(g_prof_mu);
  g_prof_on = on != 0;
  return BG_OK;
}

extern "C" int bg_profile_read(int32_t kid, double* ms_total, int64_t* launches, int32_t reset) {
  if (kid < 0 || kid >= BG_KID_COUNT) return bg_fail(BG_EINVAL, "bad kernel id");
  std::lock_guard<std::mutex> g(g_prof_mu);
  // every pending pair is read (when it can be) and destroyed exactly once, then dropped
  bool failed = false;
  for (auto& e : g_prof_events) {
    float ms = 0.f;
    if (!failed && cudaEventSynchronize(e.b) == cudaSuccess &&
        cudaEventElapsedTime(&ms, e.a, e.b) == cudaSuccess) {
      g_prof_ms[e.kid] += ms;
      g_prof_n[e.kid] += 1;
    } else {
      failed = true;
    }
    cudaEventDestroy(e.a);
    cudaEventDestroy(e.b);
  }
  g_prof_events.clear();
  if (failed) return bg_fail(BG_ECUDA, "event timing failed");
  if (ms_total) *ms_total = g_prof_ms[kid];
  if (launches) *launches = g_prof_n[kid];
  if (reset) {
    g_prof_ms[kid] = 0;
    g_prof_n[kid] = 0;
  }
  return BG_OK;
}

// ---------------------------------------------------------------------------------- status word
namespace {
std::mutex g_status_mu;
int* g_status[64] = {nullptr};

int status_word_ptr(int** out) {
  int dev = 0;
  BG_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 64) return bg_fail(BG_EINVAL, "device index out of range");
  std::lock_guard<std::mutex> g(g_status_mu);
  if (!g_status[dev]) {
    BG_CUDA(cudaMalloc(&g_status[dev], 256));
    BG_CUDA(cudaMemset(g_status[dev], 0, 256));
  }
  *out = g_status[dev];
  return BG_OK;
}
}  // namespace

int* bg_status_word_if_created(int dev) {
  if (dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> g(g_status_mu);
  return g_status[dev];
}

extern "C" int bg_selftest_device_wait(void* stream) {
  bg_clear_error();
  int* d = nullptr;
  BG_TRY(status_word_ptr(&d));
  BG_CUDA(bg::wait_selftest(d, static_cast<cudaStream_t>(stream)));
  return BG_OK;
}

extern "C" int bg_check_device(void* stream) {
  int* d = nullptr;
  BG_TRY(status_word_ptr(&d));
  cudaStream_t st = (cudaStream_t)stream;
  int h[4] = {0, 0, 0, 0};
  BG_CUDA(cudaStreamSynchronize(st));
  BG_CUDA(cudaMemcpy(h, d, sizeof(h), cudaMemcpyDeviceToHost));
  if (h[0] == 0) return BG_OK;
  BG_CUDA(cudaMemset(d, 0, 256));
  if (h[0] == 1)
    return bg_fail(BG_ETIMEOUT, "device wait gave up (kernel site " + std::to_string(h[1]) + ")");
  return bg_fail(BG_EDEVICE, "device check failed (code " + std::to_string(h[0]) + ", site " +
                                 std::to_string(h[1]) + ")");
}

// ---------------------------------------------------------------------------------- plan
extern "C" int bg_band_plan(const bg_graph* graphs, int32_t n_graphs, int32_t n_types,
                            int32_t block_S, int32_t capacity_blocks, uint32_t flags,
                            bg_plan** out) {
  bg_clear_error();
  if (flags & BG_SUPERNODES) return bg_fail(BG_EINVAL, "supernodes need bg_band_plan_opts");
  try {
    return bg_plan_build(graphs, n_graphs, n_types, block_S, capacity_blocks, flags, 0, 0, out);
  } catch (const std::bad_alloc&) {
    return bg_fail(BG_ENOMEM, "host allocation failed");
  }
}

extern "C" int bg_band_plan_opts(const bg_graph* graphs, int32_t n_graphs, int32_t n_types,
                                 int32_t block_S, int32_t capacity_blocks, const bg_plan_opts* opts,
                                 bg_plan** out) {
  bg_clear_error();
  if (!opts) return bg_fail(BG_EINVAL, "opts is NULL");
  try {
    return bg_plan_build(graphs, n_graphs, n_types, block_S, capacity_blocks, opts->flags,
                         opts->supernode_min_degree, opts->max_supernodes, out);
  } catch (const std::bad_alloc&) {
    return bg_fail(BG_ENOMEM, "host allocation failed");
  }
}

extern "C" int bg_plan_partition(const bg_plan* full, int32_t n_parts, int32_t part,
                                 bg_plan** out, bg_part_info* info) {
  bg_clear_error();
  try {
    return bg_plan_partition_build(full, n_parts, part, out, info);
  } catch (const std::bad_alloc&) {
    return bg_fail(BG_ENOMEM, "host allocation failed");
  }
}

static void free_device(bg_plan* p) {
  if (p->device < 0) return;
  int prev = 0;
  cudaGetDevice(&prev);
  cudaSetDevice(p->device);
  cudaFree(p->d_masks);
  cudaFree(p->d_masksT);
  cudaFree(p->d_gather);
  cudaFree(p->d_seg_off);
  cudaFree(p->d_seg_cnt);
  cudaFree(p->d_row_graph);
  bg::band_tc_release(p);
  bg::super_release(p);
  cudaSetDevice(prev);
  p->d_masks = p->d_masksT = nullptr;
  p->d_gather = p->d_seg_off = p->d_seg_cnt = p->d_row_graph = nullptr;
  p->device = -1;
}

extern "C" void bg_plan_free(bg_plan* plan) {
  if (!plan) return;
  free_device(plan);
  delete plan;
}

extern "C" int bg_plan_info(const bg_plan* p, bg_info* o) {
  if (!p || !o) return bg_fail(BG_EINVAL, "NULL argument");
  o->K = p->K; o->S = p->S; o->P = p->P; o->n_graphs = p->n_graphs; o->n_packed = p->n_packed;
  o->n_real = p->n_real; o->n_pad = p->n_pad(); o->n_edges_in = p->n_edges_in;
  o->n_edges_unique = p->n_unique; o->n_kept = p->n_kept; o->n_dropped = p->n_dropped;
  o->bw_before_max = p->bw_before_max; o->bw_after_max = p->bw_after_max;
  o->n_super = p->n_super; o->n_super_edges = p->n_super_edges();
  return BG_OK;
}

extern "C" double bg_plan_flops(const bg_plan* p, int32_t H, int32_t which) {
  if (!p) return 0.0;
  double K = p->K, S = p->S, P = p->P, n = p->n_pad(), h = H;
  switch (which) {
    case BG_FLOPS_BAND: return 2.0 * (3.0 * K - 2.0) * P * S * S * h;
    case BG_FLOPS_XFORM: return 2.0 * n * P * h * h;
    case BG_FLOPS_GRU: return 12.0 * n * h * h;
    case BG_FLOPS_NNZ: return 2.0 * h * (double)p->n_kept;
    default: return 0.0;
  }
}

extern "C" size_t bg_plan_export_bytes(const bg_plan* p, int32_t which) {
  if (!p) return 0;
  switch (which) {
    case BG_EXPORT_PERM: return p->perm.size() * 4;
    case BG_EXPORT_OFFSETS: return p->offset.size() * 4;
    case BG_EXPORT_MASKS:
    case BG_EXPORT_MASKS_T: return p->masks.size() * 4;
    case BG_EXPORT_BW: return p->bw_before.size() * 16;
    case BG_EXPORT_GATHER: return p->gather.size() * 4;
    case BG_EXPORT_SUPER_EDGES: return p->sup_edges.size() * 4;
    case BG_EXPORT_SUPER_COUNT: return p->nsup.size() * 4;
    default: return 0;
  }
}

extern "C" int bg_plan_export(const bg_plan* p, int32_t which, void* out, size_t out_bytes) {
  if (!p || !out) return bg_fail(BG_EINVAL, "NULL argument");
  size_t need = bg_plan_export_bytes(p, which);
  if (which < BG_EXPORT_PERM || which > BG_EXPORT_SUPER_COUNT)
    return bg_fail(BG_EINVAL, "unknown export kind");
  if (out_bytes < need) return bg_fail(BG_ECAPACITY, "export buffer too small");
  switch (which) {
    case BG_EXPORT_PERM: std::memcpy(out, p->perm.data(), need); break;
    case BG_EXPORT_OFFSETS: std::memcpy(out, p->offset.data(), need); break;
    // little-endian words with LSB-first bits are exactly the documented byte layout
    case BG_EXPORT_MASKS: std::memcpy(out, p->masks.data(), need); break;
    case BG_EXPORT_MASKS_T: std::memcpy(out, p->masksT.data(), need); break;
    case BG_EXPORT_BW: {
      int64_t* o = static_cast<int64_t*>(out);
      std::memcpy(o, p->bw_before.data(), p->bw_before.size() * 8);
      std::memcpy(o + p->bw_before.size(), p->bw_after.data(), p->bw_after.size() * 8);
      break;
    }
    case BG_EXPORT_GATHER: std::memcpy(out, p->gather.data(), need); break;
    case BG_EXPORT_SUPER_EDGES: std::memcpy(out, p->sup_edges.data(), need); break;
    case BG_EXPORT_SUPER_COUNT: std::memcpy(out, p->nsup.data(), need); break;
  }
  return BG_OK;
}

template <typename T>
static int upload_vec(const std::vector<T>& v, T** d, cudaStream_t st) {
  size_t bytes = std::max<size_t>(v.size() * sizeof(T), 16);
  BG_CUDA(cudaMalloc(d, bytes));
  if (!v.empty()) BG_CUDA(cudaMemcpyAsync(*d, v.data(), v.size() * sizeof(T), cudaMemcpyHostToDevice, st));
  return BG_OK;
}

extern "C" int bg_plan_upload(bg_plan* p, void* stream) {
  bg_clear_error();
  if (!p) return bg_fail(BG_EINVAL, "NULL plan");
  cudaStream_t st = (cudaStream_t)stream;
  int dev = 0;
  BG_CUDA(cudaGetDevice(&dev));
  free_device(p);
  p->device = dev;
  std::vector<int32_t> row_graph(p->n_pad(), -1);
  for (size_t g = 0; g < p->seg_off.size(); ++g)
    for (int32_t i = 0; i < p->seg_cnt[g]; ++i) row_graph[p->seg_off[g] + i] = (int32_t)g;
  int rc = BG_OK;
  if ((rc = upload_vec(p->masks, &p->d_masks, st)) != BG_OK ||
      (rc = upload_vec(p->masksT, &p->d_masksT, st)) != BG_OK ||
      (rc = upload_vec(p->gather, &p->d_gather, st)) != BG_OK ||
      (rc = upload_vec(p->seg_off, &p->d_seg_off, st)) != BG_OK ||
      (rc = upload_vec(p->seg_cnt, &p->d_seg_cnt, st)) != BG_OK ||
      (rc = upload_vec(row_graph, &p->d_row_graph, st)) != BG_OK) {
    free_device(p);
    return rc;
  }
  // host vectors must outlive the async copies
  BG_CUDA(cudaStreamSynchronize(st));
  if (bg::band_tc_upload(p, st) != 0 || bg::super_upload(p, st) != 0) {
    free_device(p);
    return bg_fail(BG_ENOMEM, "device allocation for the band tiles failed");
  }
  // everything a device call may need to create on this device is created here, so that the
  // allocation-free entry point finds it: the status word, its static scratch, the kernels
  int* status = nullptr;
  if ((rc = status_word_ptr(&status)) != BG_OK || (rc = bg_noalloc_prepare(p)) != BG_OK) {
    free_device(p);
    return rc;
  }
  return BG_OK;
}

// ---------------------------------------------------------------------------------- checks
static bool misaligned(const void* p) { return ((uintptr_t)p & 15u) != 0; }

static int check_plan_dev(const bg_plan* p) {
  if (!p) return bg_fail(BG_EINVAL, "NULL plan");
  if (p->device < 0 || !p->d_masks) return bg_fail(BG_ESTATE, "plan not uploaded");
  int dev = 0;
  BG_CUDA(cudaGetDevice(&dev));
  if (dev != p->device) return bg_fail(BG_ESTATE, "plan was uploaded to another device");
  return BG_OK;
}

static int check_shape(const bg_plan* p, bg_dtype dt, int32_t H) {
  if (dt != BG_F32 && dt != BG_BF16) return bg_fail(BG_EINVAL, "unknown dtype");
  if (H < 32 || H > 256 || H % 32) return bg_fail(BG_EINVAL, "H must be a multiple of 32 in [32, 256]");
  (void)p;
  return BG_OK;
}

#define BG_PTR(p, name)                                                             \
  do {                                                                              \
    if (!(p)) return bg_fail(BG_EINVAL, std::string(name) + " is NULL");            \
    if (misaligned(p)) return bg_fail(BG_EINVAL, std::string(name) + " not 16-byte aligned"); \
  } while (0)
#define BG_OPT_PTR(p, name)                                                          \
  do {                                                                              \
    if ((p) && misaligned(p)) return bg_fail(BG_EINVAL, std::string(name) + " not 16-byte aligned"); \
  } while (0)

// ---------------------------------------------------------------------------------- workspace
namespace {
inline size_t al(size_t x) { return (x + 255) & ~(size_t)255; }
inline size_t esz(bg_dtype dt) { return dt == BG_BF16 ? 2 : 4; }

// Scratch for the split-K partial sums of the small reductions.
size_t part_floats(const bg_plan* p, int H) {
  size_t a = (size_t)64 * p->P * H * H, b = (size_t)64 * 3 * H * H;
  size_t c = (size_t)256 * std::max<size_t>((size_t)p->P * H, 3 * (size_t)H);
  return std::max(std::max(a, b), c);
}

struct FwdWs {
  size_t M, band, total;
};
FwdWs fwd_ws(const bg_plan* p, bg_dtype dt, int H) {
  FwdWs w{};
  size_t n = (size_t)p->n_pad();
  w.M = 0;
  size_t band = bg::band_tc_fwd_ws_bytes(p, (int)dt, H);
  size_t simt = al(sizeof(float) * (size_t)p->P * n * H) + al((size_t)p->P * H * H * 2);
  w.band = 0;
  w.total = std::max(band, simt);
  return w;
}

// bf16 shapes the fused kernels do not cover still run their products on the tensor cores (the
// band sums stay SIMT gathers over the bit tiles); the split-K gradient GEMM needs H <= 128.
// bf16 shapes whose GEMMs run on the tensor cores: the split-K weight-gradient GEMM takes
// Hout in {32, 64, 128, 256}; other multiples of 32 use the SIMT GEMMs.
bool tc_gemm_path(bg_dtype dt, int H) {
  return dt == BG_BF16 && (H == 32 || H == 64 || H == 128 || H == 256);
}

struct BwdWs {
  size_t dM, Wt, part;                 // fp32 SIMT path
  size_t dMb, dMT, Wp, ETa, tpart;     // bf16 path with tensor-core GEMMs
  size_t super;                        // supernode edges (after everything else)
  size_t total;
};
BwdWs bwd_ws(const bg_plan* p, bg_dtype dt, int H) {
  BwdWs w{};
  size_t n = (size_t)p->n_pad();
  size_t o = 0;
  w.dM = o; o += al(sizeof(float) * n * p->P * H);
  w.Wt = o; o += al(sizeof(float) * (size_t)p->P * H * H);
  w.part = o; o += al(sizeof(float) * part_floats(p, H));
  size_t total = o;
  if (tc_gemm_path(dt, H)) {
    size_t q = 0;
    w.dMb = q; q += al(n * p->P * H * 2);
    w.dMT = q; q += al(n * p->P * H * 2);
    w.Wp = q; q += al((size_t)p->P * H * H * 2);
    w.ETa = q; q += al((size_t)(H + 16) * n * 2);
    w.tpart = q; q += al(sizeof(float) * bg::gemm_tn_part_floats(p->P * H, H + 16, (int64_t)n));
    total = std::max(total, q);
  }
  w.total = std::max(total, bg::band_tc_bwd_ws_bytes(p, (int)dt, H));
  w.super = al(w.total);
  w.total = w.super + bg::super_bwd_ws_bytes(p, H);
  return w;
}

// The GEMM-path GGNN steps of a shape whose band runs on the tensor cores and whose GRU forward
// has a fused kernel but no fused backward (bf16, H = 256): the band kernel writes Y in bf16 and
// the fused GRU forward reads it; Y is saved in bf16 (in the fp32 slot) for the backward.
bool y_bf16_path(const bg_plan* p, bg_dtype dt, int H) {
  return dt == BG_BF16 && tc_gemm_path(dt, H) && !bg::gru_tc_supported(H) &&
         bg::gru_fwd_tc_supported(H) && bg::band_tc_supported(p, (int)dt, H);
}

struct GgnnFwdWs {
  size_t gi, gh, Ybf, prop, part, addend, total;
};
GgnnFwdWs ggnn_fwd_ws(const bg_plan* p, bg_dtype dt, int H) {
  GgnnFwdWs w{};
  size_t n = (size_t)p->n_pad();
  size_t o = 0;
  w.gi = o; o += al(sizeof(float) * n * 3 * H);
  w.gh = o; o += al(sizeof(float) * n * 3 * H);
  w.Ybf = o; o += al(n * H * 2);
  w.part = o; o += al(sizeof(float) * part_floats(p, H));
  w.prop = o; o += al(fwd_ws(p, dt, H).total);
  w.addend = o; o += al(sizeof(float) * (size_t)p->sup_rows_in * H);
  w.total = o;
  return w;
}

struct GgnnBwdWs {
  size_t gi, gh, dgi, dgh, dX, g, part, prop;
  size_t Ybf, dgib, dghb, dgiT, dghT, YTa, ETa, WihT, WhhT, tpart;  // tensor-core GEMM path
  size_t dXT, dMT, Wk, tcpart, split, sup, dWs, dbs;  // and with the band kernel (bf16 Y saved)
  size_t total;
};
size_t tc_part_floats(const bg_plan* p, int H, int T);
// The GRU weight gradients of the GEMM path are reduced once over all T steps: the gate gradients
// and the Y^T, E^T operands of every step are kept side by side, [rows][T n]; the GEMM appends a
// ones row to its operand (the bias-gradient column H of a product of width H + 16).
size_t gru_tpart_floats(const bg_plan* p, int H, int T) {
  return bg::gemm_tn_part_floats(6 * H, H + 16, (int64_t)T * p->n_pad());
}
GgnnBwdWs ggnn_bwd_ws(const bg_plan* p, bg_dtype dt, int H, int T) {
  GgnnBwdWs w{};
  size_t n = (size_t)p->n_pad(), TN = (size_t)T * n;
  size_t o = 0;
  if (tc_gemm_path(dt, H)) {
    const bool ybf = y_bf16_path(p, dt, H);
    w.Ybf = o; o += al(n * H * 2);
    w.dgib = o; o += al(n * 3 * H * 2);
    w.dghb = o; o += al(n * 3 * H * 2);
    w.dgiT = o; o += al(TN * 3 * H * 2);
    w.dghT = o; o += al(TN * 3 * H * 2);
    // with the band kernel the forward keeps Y^T and E^T among the saved activations
    w.YTa = o; o += ybf ? 0 : al((size_t)(H + 16) * TN * 2);
    w.ETa = o; o += ybf ? 0 : al((size_t)(H + 16) * TN * 2);
    w.WihT = o; o += al((size_t)3 * H * H * 2);
    w.WhhT = o; o += al((size_t)3 * H * H * 2);
    w.tpart = o; o += al(sizeof(float) * gru_tpart_floats(p, H, T));
    if (ybf) {
      w.dXT = o; o += al(n * H * 2);
      w.dMT = o; o += al((size_t)p->P * H * n * 2);
      w.Wk = o; o += bg::band_tc_w_bytes(p, H);
      w.tcpart = o; o += al(sizeof(float) * tc_part_floats(p, H, T));
      w.split = o; o += al(sizeof(float) * bg::band_tc_split_floats(p, H));
      const bool sup = p->n_super_edges() > 0;
      w.sup = o; o += bg::super_bwd_ws_bytes(p, H);
      w.dWs = o; o += sup ? al(sizeof(float) * (size_t)p->P * H * H) : 0;
      w.dbs = o; o += sup ? al(sizeof(float) * (size_t)p->P * H) : 0;
    }
  }
  w.gi = o; o += al(sizeof(float) * n * 3 * H);
  w.gh = o; o += al(sizeof(float) * n * 3 * H);
  w.dgi = o; o += al(sizeof(float) * n * 3 * H);
  w.dgh = o; o += al(sizeof(float) * n * 3 * H);
  w.dX = o; o += al(sizeof(float) * n * H);
  w.g = o; o += al(sizeof(float) * n * H);
  w.part = o; o += al(sizeof(float) * part_floats(p, H));
  w.prop = o; o += al(bwd_ws(p, dt, H).total);
  w.total = o;
  return w;
}

size_t saved_E_off(const bg_plan* p, bg_dtype dt, int H, int t) {
  return (size_t)t * al(esz(dt) * (size_t)p->n_pad() * H);
}
size_t saved_Y_off(const bg_plan* p, bg_dtype dt, int H, int T, int t) {
  return saved_E_off(p, dt, H, T + 1) + (size_t)t * al(sizeof(float) * (size_t)p->n_pad() * H);
}
// With the band kernel and bf16 Y (H = 256): after E(0..T) and Y(0..T-1), E(0..T-1)^T and
// Y(0..T-1)^T in [H+16][T n] bf16 arrays, written by the forward's GRU and band kernels: the band
// products' operands and the weight-gradient GEMMs', which read the first H rows and append the
// ones row (-> bias gradient) in shared memory; the last 16 rows are not written.
struct YbSaved {
  size_t ETa, YTa, total;
};
YbSaved yb_saved(const bg_plan* p, bg_dtype dt, int H, int T) {
  const size_t TN = (size_t)T * p->n_pad();
  YbSaved s{};
  size_t o = saved_Y_off(p, dt, H, T, T);
  s.ETa = o; o += al((size_t)(H + 16) * TN * 2);
  s.YTa = o; o += al((size_t)(H + 16) * TN * 2);
  s.total = o;
  return s;
}

// ---- fused tensor-core GGNN steps (bf16, H in {32, 64, 128}, P <= 32)
// Shapes of the fused GGNN path (tensor-core band and GRU kernels): bf16, H in {32, 64, 128},
// P <= 32, a block size the band kernel has, whole 128-row tiles.
bool tc_shape(const bg_plan* p, bg_dtype dt, int H) {
  return p && dt == BG_BF16 && (H == 32 || H == 64 || H == 128) && p->P <= 32 &&
         (p->S == 32 || p->S == 64 || p->S == 128 || p->S == 256) && p->n_pad() % 128 == 0;
}
bool tc_ggnn(const bg_plan* p, bg_dtype dt, int H) {
  return tc_shape(p, dt, H) && bg::band_tc_supported(p, (int)dt, H) && bg::gru_tc_supported(H);
}

// Saved activations: E(0..T) [n][H]; E(0..T-1)^T in an [H+16][T n] array; Y(0..T-1) [n][H];
// Y(0..T-1)^T in an [H+16][T n] array (all bf16).  The transposed copies are the operands of the
// band products (TMA, K contiguous) and of the weight-gradient GEMMs, which append the ones row
// (-> bias gradient) in shared memory; the last 16 rows of each array are not written.
struct TcSaved {
  size_t E, ETa, Y, YTa, total;
};
TcSaved tc_saved(const bg_plan* p, int H, int T) {
  const size_t n = (size_t)p->n_pad(), TN = (size_t)T * n, st = al(n * H * 2);
  TcSaved s{};
  size_t o = 0;
  s.E = o; o += (size_t)(T + 1) * st;
  s.ETa = o; o += al((size_t)(H + 16) * TN * 2);
  s.Y = o; o += (size_t)T * st;
  s.YTa = o; o += al((size_t)(H + 16) * TN * 2);
  s.total = o;
  return s;
}
struct TcFwdWs {
  size_t WT, b2T, split, addend, total;
};
TcFwdWs tc_fwd_ws(const bg_plan* p, int H) {
  TcFwdWs w{};
  size_t o = 0;
  w.WT = o; o += bg::band_tc_w_bytes(p, H);
  w.b2T = o; o += al((size_t)H * 64 * 2);
  w.split = o; o += al(sizeof(float) * bg::band_tc_split_floats(p, H));
  w.addend = o; o += al(sizeof(float) * (size_t)p->sup_rows_in * H);
  w.total = o;
  return w;
}
struct TcBwdWs {
  size_t g, dXT, dMT, dgiT, dhnT, WihT, WhhT, Wk, part, split, sup, dWs, dbs, total;
};
size_t tc_part_floats(const bg_plan* p, int H, int T) {
  const int64_t K = (int64_t)T * p->n_pad();
  return std::max({bg::gemm_tn_part_floats(p->P * H, H + 16, K),
                   bg::gemm_tn_part_floats(3 * H, H + 16, K),
                   bg::gemm_tn_part_floats(p->P * H + 6 * H, H + 16, K)});
}
TcBwdWs tc_bwd_ws(const bg_plan* p, int H, int T) {
  const size_t n = (size_t)p->n_pad(), TN = (size_t)T * n;
  TcBwdWs w{};
  size_t o = 0;
  w.g = o; o += al(sizeof(float) * n * H);
  w.dXT = o; o += al(n * H * 2);
  w.dMT = o; o += al((size_t)p->P * H * TN * 2);
  w.dgiT = o; o += al((size_t)3 * H * TN * 2);
  w.dhnT = o; o += al((size_t)H * TN * 2);
  w.WihT = o; o += al((size_t)3 * H * H * 2);
  w.WhhT = o; o += al((size_t)3 * H * H * 2);
  w.Wk = o; o += bg::band_tc_w_bytes(p, H);
  w.part = o; o += al(sizeof(float) * tc_part_floats(p, H, T));
  w.split = o; o += al(sizeof(float) * bg::band_tc_split_floats(p, H));
  const bool sup = p->n_super_edges() > 0;
  w.sup = o; o += bg::super_bwd_ws_bytes(p, H);
  w.dWs = o; o += sup ? al(sizeof(float) * (size_t)p->P * H * H) : 0;
  w.dbs = o; o += sup ? al(sizeof(float) * (size_t)p->P * H) : 0;
  w.total = o;
  return w;
}
}  // namespace

extern "C" size_t bg_workspace_bytes(const bg_plan* p, bg_dtype dt, int32_t H, int32_t op) {
  if (!p || H <= 0) return 0;
  switch (op) {
    case BG_OP_PROPAGATE_FWD: return fwd_ws(p, dt, H).total;
    case BG_OP_PROPAGATE_BWD: return bwd_ws(p, dt, H).total;
    case BG_OP_READOUT:
      return al(sizeof(float) * ((size_t)p->n_packed * H + p->n_packed + 64)) +
             al(sizeof(float) * (size_t)p->n_packed * bg::kPoolSplit * H);
    default: return 0;
  }
}

extern "C" size_t bg_ggnn_workspace_bytes(const bg_plan* p, bg_dtype dt, int32_t H, int32_t T,
                                          int32_t op) {
  if (!p || H <= 0 || T < 1) return 0;
  const bool tc = tc_shape(p, dt, H);
  if (op == BG_OP_GGNN_FWD) return std::max(ggnn_fwd_ws(p, dt, H).total, tc ? tc_fwd_ws(p, H).total : 0);
  if (op == BG_OP_GGNN_BWD) return std::max(ggnn_bwd_ws(p, dt, H, T).total, tc ? tc_bwd_ws(p, H, T).total : 0);
  return 0;
}

extern "C" size_t bg_ggnn_saved_bytes(const bg_plan* p, bg_dtype dt, int32_t H, int32_t T) {
  if (!p || H <= 0 || T < 0) return 0;
  const size_t simt = saved_Y_off(p, dt, H, T, T);
  if (T >= 1 && y_bf16_path(p, dt, H)) return yb_saved(p, dt, H, T).total;
  return tc_shape(p, dt, H) && T >= 1 ? std::max(simt, tc_saved(p, H, T).total) : simt;
}

extern "C" int bg_band_uses_tensor_cores(const bg_plan* p, bg_dtype dt, int32_t H) {
  bg_clear_error();
  BG_TRY(check_plan_dev(p));
  BG_TRY(check_shape(p, dt, H));
  return bg::band_tc_supported(p, (int)dt, H) ? 1 : 0;
}

// ---------------------------------------------------------------------------------- pack
extern "C" int bg_pack_states(const bg_plan* p, bg_dtype dt, int32_t H, const void* Eo, void* Eb,
                              void* stream) {
  bg_clear_error();
  BG_TRY(check_plan_dev(p));
  if (dt != BG_F32 && dt != BG_BF16) return bg_fail(BG_EINVAL, "unknown dtype");
  if (H < 1 || H > 4096) return bg_fail(BG_EINVAL, "bad H");
  BG_PTR(Eb, "E_band");
  if (p->n_real > 0) BG_PTR(Eo, "E_orig");
  BG_CUDA(bg::pack_states(dt == BG_BF16, Eo, Eb, p->d_gather, p->n_real, p->n_pad(), H,
                          (cudaStream_t)stream));
  return BG_OK;
}

extern "C" int bg_unpack_states(const bg_plan* p, bg_dtype dt, int32_t H, const void* Eb, void* Eo,
                                void* stream) {
  bg_clear_error();
  BG_TRY(check_plan_dev(p));
  if (dt != BG_F32 && dt != BG_BF16) return bg_fail(BG_EINVAL, "unknown dtype");
  if (H < 1 || H > 4096) return bg_fail(BG_EINVAL, "bad H");
  BG_PTR(Eb, "E_band");
  BG_PTR(Eo, "E_orig");
  BG_CUDA(bg::unpack_states(dt == BG_BF16, Eb, Eo, p->d_gather, p->n_real, H, (cudaStream_t)stream));
  return BG_OK;
}

// ---------------------------------------------------------------------------------- propagate
static int propagate_fwd_impl(const bg_plan* p, bg_dtype dt, int H, const void* E, const void* W,
                              const float* b, float* Y, char* ws, size_t ws_bytes,
                              cudaStream_t st) {
  const int bf = dt == BG_BF16;
  if (bg::band_tc_supported(p, (int)dt, H)) {
    int* status = nullptr;
    BG_TRY(status_word_ptr(&status));
    // the band kernel alone is timed inside (its operand preparation is not)
    BG_CUDA(bg::band_tc_fwd(p, H, E, W, b, Y, ws, ws_bytes, status, st));
    // the supernode rows and columns (Section 6), added to the band's sums
    BG_CUDA(bg::super_fwd(p, bf, H, E, W, b, Y, 0, st));
    return BG_OK;
  }
  // SIMT path: messages M_p = E W_p + b_p for all p, then the band sum over the bit tiles
  const size_t n = (size_t)p->n_pad();
  float* M = reinterpret_cast<float*>(ws);
  if (ws_bytes < sizeof(float) * (size_t)p->P * n * H) return bg_fail(BG_ECAPACITY, "workspace too small");
  KTimer t(BG_KID_BAND_FWD, st);
  if (bf) {
    // transforms on the tensor cores: M_p = E W_p + b_p with W_p^T as the K-major operand
    int* status = nullptr;
    BG_TRY(status_word_ptr(&status));
    auto* WT = reinterpret_cast<__nv_bfloat16*>(ws + al(sizeof(float) * (size_t)p->P * n * H));
    BG_CUDA(bg::prep_transpose_bf16(W, 0, WT, H, H, p->P, st));
    BG_CUDA(bg::gemm_bf16_tn(E, H, 0, WT, H, (int64_t)H * H, (int)n, H, H, p->P, M, H,
                             (int64_t)n * H, b, H, 0, status, st));
  } else {
    bg::Gemm g;
    g.M = (int)n; g.N = H; g.K = H; g.batch = p->P;
    g.A = E; g.a_bf16 = bf; g.sAb = 0; g.sAm = H; g.sAk = 1;
    g.B = W; g.b_bf16 = bf; g.sBb = (int64_t)H * H; g.sBk = H; g.sBn = 1;
    g.C = M; g.sCb = (int64_t)n * H; g.ldc = H;
    g.bias = b; g.sBias = H;
    BG_CUDA(bg::gemm(g, nullptr, 0, st));
  }
  BG_CUDA(bg::band_fwd_gather(p->d_masks, M, Y, p->K, p->S, p->P, H, st));
  BG_CUDA(bg::super_fwd(p, bf, H, E, W, b, Y, 0, st));
  return BG_OK;
}

extern "C" int bg_band_propagate_fwd(const bg_plan* p, bg_dtype dt, int32_t H, const void* E,
                                     const void* W, const float* b, float* Y, void* ws,
                                     size_t ws_bytes, void* stream) {
  bg_clear_error();
  BG_TRY(check_plan_dev(p));
  BG_TRY(check_shape(p, dt, H));
  BG_PTR(E, "E"); BG_PTR(W, "W"); BG_OPT_PTR(b, "b"); BG_PTR(Y, "Y"); BG_PTR(ws, "ws");
  if (ws_bytes < fwd_ws(p, dt, H).total) return bg_fail(BG_ECAPACITY, "workspace too small");
  return propagate_fwd_impl(p, dt, H, E, W, b, Y, static_cast<char*>(ws), ws_bytes,
                            (cudaStream_t)stream);
}

static int propagate_bwd_band(const bg_plan* p, bg_dtype dt, int H, const void* E, const void* W,
                              const float* dY, float* dE, float* dW, float* db, int accum,
                              char* ws, size_t ws_bytes, cudaStream_t st);

// dE/dW/db accumulate when accum != 0 (callers zero them first otherwise).
static int propagate_bwd_impl(const bg_plan* p, bg_dtype dt, int H, const void* E, const void* W,
                              const float* dY, float* dE, float* dW, float* db, int accum,
                              char* ws, size_t ws_bytes, cudaStream_t st) {
  const int bf = dt == BG_BF16;
  BwdWs w = bwd_ws(p, dt, H);
  if (ws_bytes < w.total) return bg_fail(BG_ECAPACITY, "workspace too small");
  BG_TRY(propagate_bwd_band(p, dt, H, E, W, dY, dE, dW, db, accum, ws, ws_bytes, st));
  // the supernode rows and columns (Section 6), added to the band's gradients
  BG_CUDA(bg::super_bwd(p, bf, H, E, W, dY, nullptr, 0, dE, dW, db, ws + w.super, st));
  return BG_OK;
}

// The band part of propagate_bwd_impl.
static int propagate_bwd_band(const bg_plan* p, bg_dtype dt, int H, const void* E, const void* W,
                              const float* dY, float* dE, float* dW, float* db, int accum,
                              char* ws, size_t ws_bytes, cudaStream_t st) {
  const int bf = dt == BG_BF16;
  const size_t n = (size_t)p->n_pad();
  if (bg::band_tc_supported(p, (int)dt, H)) {
    int* status = nullptr;
    BG_TRY(status_word_ptr(&status));
    // the band kernel and the weight-gradient GEMM are timed inside
    BG_CUDA(bg::band_tc_bwd(p, H, E, W, dY, dE, dW, db, accum, ws, ws_bytes, status, st));
    return BG_OK;
  }
  BwdWs w = bwd_ws(p, dt, H);
  if (tc_gemm_path(dt, H)) {
    int* status = nullptr;
    BG_TRY(status_word_ptr(&status));
    auto* dMb = reinterpret_cast<__nv_bfloat16*>(ws + w.dMb);
    auto* dMT = reinterpret_cast<__nv_bfloat16*>(ws + w.dMT);
    auto* Wp = reinterpret_cast<__nv_bfloat16*>(ws + w.Wp);
    auto* ETa = reinterpret_cast<__nv_bfloat16*>(ws + w.ETa);
    float* tpart = reinterpret_cast<float*>(ws + w.tpart);
    const size_t tpf = bg::gemm_tn_part_floats(p->P * H, H + 16, (int64_t)n);
    const int PH = p->P * H;
    {
      KTimer t(BG_KID_BAND_BWD, st);
      // dM_p = A_p^T dY over the transposed bit tiles; dE (+)= dM_cat [n][P*H] x Wp^T
      BG_CUDA(bg::band_bwd_gather_bf16(p->d_masksT, dY, dMb, p->K, p->S, p->P, H, st));
      BG_CUDA(bg::wperm(W, Wp, p->P, H, st));
      BG_CUDA(bg::gemm_bf16_tn(dMb, PH, 0, Wp, PH, 0, (int)n, H, PH, 1, dE, H, 0, nullptr, 0,
                               accum, status, st));
    }
    KTimer t(BG_KID_DW, st);
    // dW_p, db_p from one split-K product of dM^T with E^T and the GEMM's appended ones row
    BG_CUDA(bg::prep_transpose_bf16(dMb, 0, dMT, (int)n, PH, 1, st));
    BG_CUDA(bg::prep_transpose_bf16(E, 0, ETa, (int)n, H, 1, st));
    BG_CUDA(bg::gemm_tn(dMT, (int64_t)n, ETa, (int64_t)n, PH, H, (int64_t)n, 1, dW, db, accum,
                        tpart, tpf, status, st));
    return BG_OK;
  }
  float* dM = reinterpret_cast<float*>(ws + w.dM);
  float* Wt = reinterpret_cast<float*>(ws + w.Wt);
  float* part = reinterpret_cast<float*>(ws + w.part);
  const size_t pf = part_floats(p, H);
  {
    KTimer t(BG_KID_BAND_BWD, st);
    BG_CUDA(bg::band_bwd_gather(p->d_masksT, dY, dM, p->K, p->S, p->P, H, st));
    // dE (+)= dM_cat [n, P*H] x Wt_cat [P*H, H]
    BG_CUDA(bg::transpose_weights(bf, W, Wt, p->P, H, st));
    bg::Gemm g;
    g.M = (int)n; g.N = H; g.K = p->P * H;
    g.A = dM; g.sAm = (int64_t)p->P * H; g.sAk = 1;
    g.B = Wt; g.sBk = H; g.sBn = 1;
    g.C = dE; g.ldc = H; g.accumulate = accum;
    BG_CUDA(bg::gemm(g, part, pf, st));
  }
  {
    KTimer t(BG_KID_DW, st);
    // dW_p (+)= E^T dM_p
    bg::Gemm g;
    g.M = H; g.N = H; g.K = (int)n; g.batch = p->P;
    g.A = E; g.a_bf16 = bf; g.sAb = 0; g.sAm = 1; g.sAk = H;
    g.B = dM; g.sBb = H; g.sBk = (int64_t)p->P * H; g.sBn = 1;
    g.C = dW; g.sCb = (int64_t)H * H; g.ldc = H; g.accumulate = accum;
    BG_CUDA(bg::gemm(g, part, pf, st));
    if (db) BG_CUDA(bg::colsum(dM, (int64_t)n, p->P * H, db, accum, part, pf, st));
  }
  return BG_OK;
}

extern "C" int bg_band_propagate_bwd(const bg_plan* p, bg_dtype dt, int32_t H, const void* E,
                                     const void* W, const float* dY, float* dE, float* dW,
                                     float* db, uint32_t flags, void* ws, size_t ws_bytes,
                                     void* stream) {
  bg_clear_error();
  BG_TRY(check_plan_dev(p));
  BG_TRY(check_shape(p, dt, H));
  BG_PTR(E, "E"); BG_PTR(W, "W"); BG_PTR(dY, "dY"); BG_PTR(dE, "dE"); BG_PTR(dW, "dW");
  BG_OPT_PTR(db, "db"); BG_PTR(ws, "ws");
  if (ws_bytes < bwd_ws(p, dt, H).total) return bg_fail(BG_ECAPACITY, "workspace too small");
  return propagate_bwd_impl(p, dt, H, E, W, dY, dE, dW, db, (flags & BG_ACCUM) ? 1 : 0,
                            static_cast<char*>(ws), ws_bytes, (cudaStream_t)stream);
}

// ---------------------------------------------------------------------------------- GGNN
static int check_params(const bg_params* prm) {
  if (!prm) return bg_fail(BG_EINVAL, "params is NULL");
  BG_PTR(prm->W, "W"); BG_OPT_PTR(prm->b, "b"); BG_PTR(prm->W_ih, "W_ih");
  BG_PTR(prm->W_hh, "W_hh"); BG_PTR(prm->b_ih, "b_ih"); BG_PTR(prm->b_hh, "b_hh");
  return BG_OK;
}

// gi = X W_ih^T + b_ih, gh = Hs W_hh^T + b_hh  ([n, 3H] fp32).  With Xb (bf16 scratch [n][H]) the
// products run on the tensor cores (W_ih, W_hh are already K-major [3H][H] operands); X NULL means
// Xb already holds the messages in bf16.
static int gru_gates_in(const bg_plan* p, int bf, int H, const float* X, const void* Hs,
                        const bg_params* prm, float* gi, float* gh, float* part, size_t pf,
                        cudaStream_t st, __nv_bfloat16* Xb = nullptr) {
  const int n = p->n_pad();
  if (Xb) {
    int* status = nullptr;
    BG_TRY(status_word_ptr(&status));
    if (X) BG_CUDA(bg::f32_to_bf16(X, Xb, (int64_t)n * H, st));
    BG_CUDA(bg::gemm_bf16_tn(Xb, H, 0, prm->W_ih, H, 0, n, 3 * H, H, 1, gi, 3 * H, 0, prm->b_ih, 0,
                             0, status, st));
    BG_CUDA(bg::gemm_bf16_tn(Hs, H, 0, prm->W_hh, H, 0, n, 3 * H, H, 1, gh, 3 * H, 0, prm->b_hh, 0,
                             0, status, st));
    return BG_OK;
  }
  bg::Gemm g;
  g.M = n; g.N = 3 * H; g.K = H;
  g.A = X; g.sAm = H; g.sAk = 1;
  g.B = prm->W_ih; g.b_bf16 = bf; g.sBk = 1; g.sBn = H;
  g.C = gi; g.ldc = 3 * H; g.bias = prm->b_ih;
  BG_CUDA(bg::gemm(g, part, pf, st));
  bg::Gemm h;
  h.M = n; h.N = 3 * H; h.K = H;
  h.A = Hs; h.a_bf16 = bf; h.sAm = H; h.sAk = 1;
  h.B = prm->W_hh; h.b_bf16 = bf; h.sBk = 1; h.sBn = H;
  h.C = gh; h.ldc = 3 * H; h.bias = prm->b_hh;
  BG_CUDA(bg::gemm(h, part, pf, st));
  return BG_OK;
}

extern "C" int bg_ggnn_step(const bg_plan* p, bg_dtype dt, int32_t H, int32_t T,
                            const bg_params* prm, const void* E0, void* ET, void* saved,
                            size_t saved_bytes, void* ws, size_t ws_bytes, void* stream) {
  bg_clear_error();
  BG_TRY(check_plan_dev(p));
  BG_TRY(check_shape(p, dt, H));
  BG_TRY(check_params(prm));
  if (T < 1 || T > 1024) return bg_fail(BG_EINVAL, "T must be in [1, 1024]");
  BG_PTR(E0, "E0"); BG_OPT_PTR(ET, "ET"); BG_PTR(saved, "saved"); BG_PTR(ws, "ws");
  if (saved_bytes < bg_ggnn_saved_bytes(p, dt, H, T)) return bg_fail(BG_ECAPACITY, "saved buffer too small");
  if (ws_bytes < bg_ggnn_workspace_bytes(p, dt, H, T, BG_OP_GGNN_FWD))
    return bg_fail(BG_ECAPACITY, "workspace too small");
  cudaStream_t st = (cudaStream_t)stream;
  if (tc_ggnn(p, dt, H)) {
    int* status = nullptr;
    BG_TRY(status_word_ptr(&status));
    const size_t n = (size_t)p->n_pad(), TN = (size_t)T * n, stE = al(n * H * 2);
    const TcSaved sl = tc_saved(p, H, T);
    const TcFwdWs wl = tc_fwd_ws(p, H);
    char* sv = static_cast<char*>(saved);
    char* wsc = static_cast<char*>(ws);
    auto Ei = [&](int t) { return reinterpret_cast<__nv_bfloat16*>(sv + sl.E + (size_t)t * stE); };
    auto Yi = [&](int t) { return reinterpret_cast<__nv_bfloat16*>(sv + sl.Y + (size_t)t * stE); };
    __nv_bfloat16* ETa = reinterpret_cast<__nv_bfloat16*>(sv + sl.ETa);
    __nv_bfloat16* YTa = reinterpret_cast<__nv_bfloat16*>(sv + sl.YTa);
    void* WT = wsc + wl.WT;
    __nv_bfloat16* b2T = reinterpret_cast<__nv_bfloat16*>(wsc + wl.b2T);
    float* split = bg::band_tc_split_floats(p, H) ? reinterpret_cast<float*>(wsc + wl.split)
                                                   : nullptr;
    float* addend = p->sup_rows_in ? reinterpret_cast<float*>(wsc + wl.addend) : nullptr;
    BG_CUDA(cudaMemcpyAsync(Ei(0), E0, n * H * 2, cudaMemcpyDeviceToDevice, st));
    BG_CUDA(bg::prep_transpose_bf16(E0, 0, ETa, (int)n, H, 1, st, (int64_t)TN));
    BG_CUDA(bg::band_tc_prep_w(p, H, prm->W, 0, WT, st));
    if (prm->b) BG_CUDA(bg::prep_bias_split(p, prm->b, b2T, H, status, st));
    for (int t = 0; t < T; ++t) {
      // the supernode rows' messages, which the band kernel adds before it rounds Y
      if (addend) BG_CUDA(bg::super_fwd(p, 1, H, Ei(t), prm->W, prm->b, addend, 1, st));
      {
        KTimer tm(BG_KID_BAND_FWD, st);
        BG_CUDA(bg::band_tc_fwd_core(p, H, ETa + (size_t)t * n, (int64_t)TN, WT,
                                     prm->b ? b2T : nullptr, prm->b, nullptr, Yi(t),
                                     YTa + (size_t)t * n, (int64_t)TN, split, addend, status, st));
      }
      KTimer tm(BG_KID_GRU_FWD, st);
      BG_CUDA(bg::gru_fwd_tc(
          H, (int)n, p->n_real, Yi(t), Ei(t), static_cast<const __nv_bfloat16*>(prm->W_ih),
          static_cast<const __nv_bfloat16*>(prm->W_hh), prm->b_ih, prm->b_hh, Ei(t + 1),
          t + 1 < T ? ETa + (size_t)(t + 1) * n : nullptr, (int64_t)TN, status, st));
    }
    if (ET) BG_CUDA(cudaMemcpyAsync(ET, Ei(T), n * H * 2, cudaMemcpyDeviceToDevice, st));
    return BG_OK;
  }
  GgnnFwdWs w = ggnn_fwd_ws(p, dt, H);
  const int bf = dt == BG_BF16;
  char* sv = static_cast<char*>(saved);
  char* wsc = static_cast<char*>(ws);
  float* gi = reinterpret_cast<float*>(wsc + w.gi);
  float* gh = reinterpret_cast<float*>(wsc + w.gh);
  float* part = reinterpret_cast<float*>(wsc + w.part);
  const size_t pf = part_floats(p, H);
  const size_t ebytes = esz(dt) * (size_t)p->n_pad() * H;
  BG_CUDA(cudaMemcpyAsync(sv + saved_E_off(p, dt, H, 0), E0, ebytes, cudaMemcpyDeviceToDevice, st));
  if (y_bf16_path(p, dt, H)) {
    // band kernel (bf16 Y and Y^T) and the fused GRU forward (E(t+1) and E(t+1)^T): the
    // transposed copies go to the saved E^T and Y^T arrays for the band products of the next
    // step and for the backward's weight gradients
    int* status = nullptr;
    BG_TRY(status_word_ptr(&status));
    const size_t n = (size_t)p->n_pad(), TN = (size_t)T * n;
    const YbSaved ys = yb_saved(p, dt, H, T);
    auto* ETa = reinterpret_cast<__nv_bfloat16*>(sv + ys.ETa);
    auto* YTa = reinterpret_cast<__nv_bfloat16*>(sv + ys.YTa);
    char* pw = wsc + w.prop;
    void* WT = pw + al(n * H * 2);
    auto* b2T = reinterpret_cast<__nv_bfloat16*>(pw + al(n * H * 2) + bg::band_tc_w_bytes(p, H));
    float* split = reinterpret_cast<float*>(pw + al(n * H * 2) + bg::band_tc_w_bytes(p, H) +
                                            al((size_t)H * 64 * 2));
    float* addend = p->sup_rows_in ? reinterpret_cast<float*>(wsc + w.addend) : nullptr;
    BG_CUDA(bg::prep_transpose_bf16(E0, 0, ETa, (int)n, H, 1, st, (int64_t)TN));
    BG_CUDA(bg::band_tc_prep_w(p, H, prm->W, 0, WT, st));
    if (prm->b) BG_CUDA(bg::prep_bias_split(p, prm->b, b2T, H, status, st));
    for (int t = 0; t < T; ++t) {
      const auto* Et = reinterpret_cast<const __nv_bfloat16*>(sv + saved_E_off(p, dt, H, t));
      auto* En = reinterpret_cast<__nv_bfloat16*>(sv + saved_E_off(p, dt, H, t + 1));
      auto* Yb = reinterpret_cast<__nv_bfloat16*>(sv + saved_Y_off(p, dt, H, T, t));
      if (addend) BG_CUDA(bg::super_fwd(p, 1, H, Et, prm->W, prm->b, addend, 1, st));
      {
        KTimer tm(BG_KID_BAND_FWD, st);
        BG_CUDA(bg::band_tc_fwd_core(p, H, ETa + (size_t)t * n, (int64_t)TN, WT,
                                     prm->b ? b2T : nullptr, prm->b, nullptr, Yb,
                                     YTa + (size_t)t * n, (int64_t)TN,
                                     bg::band_tc_split_floats(p, H) ? split : nullptr, addend,
                                     status, st));
      }
      KTimer tm(BG_KID_GRU_FWD, st);
      BG_CUDA(bg::gru_fwd_tc(H, (int)n, p->n_real, Yb, Et,
                             static_cast<const __nv_bfloat16*>(prm->W_ih),
                             static_cast<const __nv_bfloat16*>(prm->W_hh), prm->b_ih, prm->b_hh, En,
                             t + 1 < T ? ETa + (size_t)(t + 1) * n : nullptr, (int64_t)TN, status,
                             st));
    }
    if (ET) BG_CUDA(cudaMemcpyAsync(ET, sv + saved_E_off(p, dt, H, T), ebytes, cudaMemcpyDeviceToDevice, st));
    return BG_OK;
  }
  for (int t = 0; t < T; ++t) {
    const void* Et = sv + saved_E_off(p, dt, H, t);
    void* En = sv + saved_E_off(p, dt, H, t + 1);
    float* Yt = reinterpret_cast<float*>(sv + saved_Y_off(p, dt, H, T, t));
    BG_TRY(propagate_fwd_impl(p, dt, H, Et, prm->W, prm->b, Yt, wsc + w.prop, w.total - w.prop, st));
    KTimer tm(BG_KID_GRU_FWD, st);
    BG_TRY(gru_gates_in(p, bf, H, Yt, Et, prm, gi, gh, part, pf, st,
                        tc_gemm_path(dt, H) ? reinterpret_cast<__nv_bfloat16*>(wsc + w.Ybf)
                                            : nullptr));
    BG_CUDA(bg::gru_fwd_gates(bf, gi, gh, Et, En, p->n_real, p->n_pad(), H, st));
  }
  if (ET) BG_CUDA(cudaMemcpyAsync(ET, sv + saved_E_off(p, dt, H, T), ebytes, cudaMemcpyDeviceToDevice, st));
  return BG_OK;
}

extern "C" int bg_ggnn_step_bwd(const bg_plan* p, bg_dtype dt, int32_t H, int32_t T,
                                const bg_params* prm, const void* saved, size_t saved_bytes,
                                const float* dET, float* dE0, const bg_grads* gr, uint32_t flags,
                                void* ws, size_t ws_bytes, void* stream) {
  bg_clear_error();
  BG_TRY(check_plan_dev(p));
  BG_TRY(check_shape(p, dt, H));
  BG_TRY(check_params(prm));
  if (T < 1 || T > 1024) return bg_fail(BG_EINVAL, "T must be in [1, 1024]");
  if (!gr) return bg_fail(BG_EINVAL, "grads is NULL");
  BG_PTR(saved, "saved"); BG_PTR(dET, "dET"); BG_PTR(dE0, "dE0"); BG_PTR(ws, "ws");
  BG_PTR(gr->dW, "dW"); BG_OPT_PTR(gr->db, "db"); BG_PTR(gr->dW_ih, "dW_ih");
  BG_PTR(gr->dW_hh, "dW_hh"); BG_PTR(gr->db_ih, "db_ih"); BG_PTR(gr->db_hh, "db_hh");
  if (saved_bytes < bg_ggnn_saved_bytes(p, dt, H, T)) return bg_fail(BG_ECAPACITY, "saved buffer too small");
  if (ws_bytes < bg_ggnn_workspace_bytes(p, dt, H, T, BG_OP_GGNN_BWD))
    return bg_fail(BG_ECAPACITY, "workspace too small");
  cudaStream_t st = (cudaStream_t)stream;
  if (tc_ggnn(p, dt, H)) {
    int* status = nullptr;
    BG_TRY(status_word_ptr(&status));
    const size_t n = (size_t)p->n_pad(), TN = (size_t)T * n, stE = al(n * H * 2);
    const TcSaved sl = tc_saved(p, H, T);
    const TcBwdWs wl = tc_bwd_ws(p, H, T);
    const char* sv = static_cast<const char*>(saved);
    char* wsc = static_cast<char*>(ws);
    auto Ei = [&](int t) { return reinterpret_cast<const __nv_bfloat16*>(sv + sl.E + (size_t)t * stE); };
    auto Yi = [&](int t) { return reinterpret_cast<const __nv_bfloat16*>(sv + sl.Y + (size_t)t * stE); };
    const __nv_bfloat16* ETa = reinterpret_cast<const __nv_bfloat16*>(sv + sl.ETa);
    const __nv_bfloat16* YTa = reinterpret_cast<const __nv_bfloat16*>(sv + sl.YTa);
    float* g = reinterpret_cast<float*>(wsc + wl.g);
    __nv_bfloat16* dXT = reinterpret_cast<__nv_bfloat16*>(wsc + wl.dXT);
    __nv_bfloat16* dMT = reinterpret_cast<__nv_bfloat16*>(wsc + wl.dMT);
    __nv_bfloat16* dgiT = reinterpret_cast<__nv_bfloat16*>(wsc + wl.dgiT);
    __nv_bfloat16* dhnT = reinterpret_cast<__nv_bfloat16*>(wsc + wl.dhnT);
    __nv_bfloat16* WihT = reinterpret_cast<__nv_bfloat16*>(wsc + wl.WihT);
    __nv_bfloat16* WhhT = reinterpret_cast<__nv_bfloat16*>(wsc + wl.WhhT);
    float* part = reinterpret_cast<float*>(wsc + wl.part);
    const size_t pf = tc_part_floats(p, H, T);
    float* split = bg::band_tc_split_floats(p, H) ? reinterpret_cast<float*>(wsc + wl.split)
                                                   : nullptr;
    const auto* Wih = static_cast<const __nv_bfloat16*>(prm->W_ih);
    const auto* Whh = static_cast<const __nv_bfloat16*>(prm->W_hh);
    BG_CUDA(bg::prep_transpose_bf16(Wih, 0, WihT, 3 * H, H, 1, st));
    BG_CUDA(bg::prep_transpose_bf16(Whh, 0, WhhT, 3 * H, H, 1, st));
    void* Wk = wsc + wl.Wk;
    BG_CUDA(bg::band_tc_prep_w(p, H, prm->W, 1, Wk, st));
    const bool sup = p->n_super_edges() > 0;
    float* dWs = reinterpret_cast<float*>(wsc + wl.dWs);
    float* dbs = reinterpret_cast<float*>(wsc + wl.dbs);
    if (sup) {
      BG_CUDA(bg::fill_zero_f32(dWs, (int64_t)p->P * H * H, st));
      BG_CUDA(bg::fill_zero_f32(dbs, (int64_t)p->P * H, st));
    }
    const float* gin = dET;
    for (int t = T - 1; t >= 0; --t) {
      {
        KTimer tm(BG_KID_GRU_BWD, st);
        BG_CUDA(bg::gru_bwd_tc(H, (int)n, p->n_real, Yi(t), Ei(t), Wih, Whh, WihT, WhhT, prm->b_ih,
                               prm->b_hh, gin, g, dXT, (int64_t)n, dgiT + (size_t)t * n,
                               dhnT + (size_t)t * n, (int64_t)TN, status, st));
      }
      {
        KTimer tm(BG_KID_BAND_BWD, st);
        BG_CUDA(bg::band_tc_bwd_core(p, H, dXT, (int64_t)n, Wk, g, 1, dMT + (size_t)t * n,
                                     (int64_t)TN, split, status, st));
      }
      // the supernode rows and columns: dE(t) and their share of dW, db (summed over the steps)
      if (sup)
        BG_CUDA(bg::super_bwd(p, 1, H, Ei(t), prm->W, nullptr, dXT, (int64_t)n, g, dWs, dbs,
                              wsc + wl.sup, st, t < T - 1));
      gin = g;
    }
    const int acc = (flags & BG_ACCUM) ? 1 : 0;
    KTimer tm(BG_KID_DW, st);
    // dW_p, db_p over all steps and nodes; dW_ih, db_ih; dW_hh, db_hh, whose r and z rows take
    // the input-side gate gradients (equal to the hidden-side ones there) and n rows dh_n
    const bg::TNProblem probs[4] = {
        {dMT, (int64_t)TN, ETa, (int64_t)TN, p->P * H, 1, gr->dW, gr->db},
        {dgiT, (int64_t)TN, YTa, (int64_t)TN, 3 * H, 0, gr->dW_ih, gr->db_ih},
        {dgiT, (int64_t)TN, ETa, (int64_t)TN, 2 * H, 0, gr->dW_hh, gr->db_hh},
        {dhnT, (int64_t)TN, ETa, (int64_t)TN, H, 0, gr->dW_hh + (size_t)2 * H * H,
         gr->db_hh + 2 * H}};
    BG_CUDA(bg::gemm_tn_multi(probs, 4, H, (int64_t)TN, acc, part, pf, status, st));
    if (sup) {
      BG_CUDA(bg::add_inplace_f32(gr->dW, dWs, (int64_t)p->P * H * H, st));
      if (gr->db) BG_CUDA(bg::add_inplace_f32(gr->db, dbs, (int64_t)p->P * H, st));
    }
    BG_CUDA(cudaMemcpyAsync(dE0, g, sizeof(float) * n * H, cudaMemcpyDeviceToDevice, st));
    return BG_OK;
  }
  GgnnBwdWs w = ggnn_bwd_ws(p, dt, H, T);
  const int bf = dt == BG_BF16;
  const int n = p->n_pad();
  const char* sv = static_cast<const char*>(saved);
  char* wsc = static_cast<char*>(ws);
  float* gi = reinterpret_cast<float*>(wsc + w.gi);
  float* gh = reinterpret_cast<float*>(wsc + w.gh);
  float* dgi = reinterpret_cast<float*>(wsc + w.dgi);
  float* dgh = reinterpret_cast<float*>(wsc + w.dgh);
  float* dX = reinterpret_cast<float*>(wsc + w.dX);
  float* g = reinterpret_cast<float*>(wsc + w.g);
  float* part = reinterpret_cast<float*>(wsc + w.part);
  const size_t pf = part_floats(p, H);
  if (y_bf16_path(p, dt, H)) {
    // H = 256 with the band kernel: per step the gate gradients (one kernel), dX^T = (dgi W_ih)^T
    // straight into the band backward's operand, g += dgh W_hh, the transposed-band backward and
    // the band's weight gradients from its dM_p^T (one step's K range of E^T stays in L2
    // across the M tiles, which a product over all T steps at once does not); the GRU's weight
    // gradients in one grouped product over all T steps at the end (operands E^T, Y^T
    // saved by the forward).  The running state gradient alternates between two buffers.
    int* status = nullptr;
    BG_TRY(status_word_ptr(&status));
    const size_t nn = (size_t)n, TN = (size_t)T * nn;
    const YbSaved ys = yb_saved(p, dt, H, T);
    const auto* ETa = reinterpret_cast<const __nv_bfloat16*>(sv + ys.ETa);
    const auto* YTa = reinterpret_cast<const __nv_bfloat16*>(sv + ys.YTa);
    auto* dgib = reinterpret_cast<__nv_bfloat16*>(wsc + w.dgib);
    auto* dghb = reinterpret_cast<__nv_bfloat16*>(wsc + w.dghb);
    auto* dgiT = reinterpret_cast<__nv_bfloat16*>(wsc + w.dgiT);
    auto* dghT = reinterpret_cast<__nv_bfloat16*>(wsc + w.dghT);
    auto* WihT = reinterpret_cast<__nv_bfloat16*>(wsc + w.WihT);
    auto* WhhT = reinterpret_cast<__nv_bfloat16*>(wsc + w.WhhT);
    auto* dXT = reinterpret_cast<__nv_bfloat16*>(wsc + w.dXT);
    auto* dMT = reinterpret_cast<__nv_bfloat16*>(wsc + w.dMT);
    void* Wk = wsc + w.Wk;
    float* tcpart = reinterpret_cast<float*>(wsc + w.tcpart);
    float* split = bg::band_tc_split_floats(p, H) ? reinterpret_cast<float*>(wsc + w.split)
                                                   : nullptr;
    const auto* Wih = static_cast<const __nv_bfloat16*>(prm->W_ih);
    const auto* Whh = static_cast<const __nv_bfloat16*>(prm->W_hh);
    BG_CUDA(bg::prep_transpose_bf16(Wih, 0, WihT, 3 * H, H, 1, st));
    BG_CUDA(bg::prep_transpose_bf16(Whh, 0, WhhT, 3 * H, H, 1, st));
    BG_CUDA(bg::band_tc_prep_w(p, H, prm->W, 1, Wk, st));
    const bool sup = p->n_super_edges() > 0;
    float* dWs = reinterpret_cast<float*>(wsc + w.dWs);
    float* dbs = reinterpret_cast<float*>(wsc + w.dbs);
    if (sup) {
      BG_CUDA(bg::fill_zero_f32(dWs, (int64_t)p->P * H * H, st));
      BG_CUDA(bg::fill_zero_f32(dbs, (int64_t)p->P * H, st));
    }
    const int acc = (flags & BG_ACCUM) ? 1 : 0;
    const float* gin = dET;
    float* gout = dX;
    for (int t = T - 1; t >= 0; --t) {
      const auto* Et = reinterpret_cast<const __nv_bfloat16*>(sv + saved_E_off(p, dt, H, t));
      const auto* Yt = reinterpret_cast<const __nv_bfloat16*>(sv + saved_Y_off(p, dt, H, T, t));
      {
        KTimer tm(BG_KID_GRU_BWD, st);
        BG_CUDA(bg::gru_bwd_gates_tc(H, n, p->n_real, Yt, Et, Wih, Whh, prm->b_ih, prm->b_hh, gin,
                                     gout, dgib, dghb, dgiT + (size_t)t * nn,
                                     dghT + (size_t)t * nn, (int64_t)TN, status, st));
        BG_CUDA(bg::gemm_bf16_tn_outT(dgib, 3 * H, WihT, 3 * H, n, H, 3 * H, dXT, (int64_t)nn,
                                      status, st));
        BG_CUDA(bg::gemm_bf16_tn(dghb, 3 * H, 0, WhhT, 3 * H, 0, n, H, 3 * H, 1, gout, H, 0,
                                 nullptr, 0, 1, status, st));
      }
      {
        KTimer tm(BG_KID_BAND_BWD, st);
        BG_CUDA(bg::band_tc_bwd_core(p, H, dXT, (int64_t)nn, Wk, gout, 1, dMT, (int64_t)nn, split,
                                     status, st));
      }
      {
        KTimer tm(BG_KID_DW, st);
        BG_CUDA(bg::gemm_tn(dMT, (int64_t)nn, ETa + (size_t)t * nn, (int64_t)TN, p->P * H, H,
                            (int64_t)nn, 1, gr->dW, gr->db, t == T - 1 ? acc : 1, tcpart,
                            tc_part_floats(p, H, T), status, st));
      }
      // the supernode rows and columns: dE(t) and their share of dW, db (summed over the steps)
      if (sup)
        BG_CUDA(bg::super_bwd(p, 1, H, Et, prm->W, nullptr, dXT, (int64_t)nn, gout, dWs, dbs,
                              wsc + w.sup, st, t < T - 1));
      gin = gout;
      gout = gout == dX ? g : dX;
    }
    KTimer tm(BG_KID_DW, st);
    const bg::TNProblem probs[2] = {
        {dgiT, (int64_t)TN, YTa, (int64_t)TN, 3 * H, 0, gr->dW_ih, gr->db_ih},
        {dghT, (int64_t)TN, ETa, (int64_t)TN, 3 * H, 0, gr->dW_hh, gr->db_hh}};
    BG_CUDA(bg::gemm_tn_multi(probs, 2, H, (int64_t)TN, acc, tcpart, tc_part_floats(p, H, T),
                              status, st));
    if (sup) {
      BG_CUDA(bg::add_inplace_f32(gr->dW, dWs, (int64_t)p->P * H * H, st));
      if (gr->db) BG_CUDA(bg::add_inplace_f32(gr->db, dbs, (int64_t)p->P * H, st));
    }
    BG_CUDA(cudaMemcpyAsync(dE0, gin, sizeof(float) * nn * H, cudaMemcpyDeviceToDevice, st));
    return BG_OK;
  }
  if (!(flags & BG_ACCUM)) {
    BG_CUDA(bg::fill_zero_f32(gr->dW, (int64_t)p->P * H * H, st));
    if (gr->db) BG_CUDA(bg::fill_zero_f32(gr->db, (int64_t)p->P * H, st));
    BG_CUDA(bg::fill_zero_f32(gr->dW_ih, 3LL * H * H, st));
    BG_CUDA(bg::fill_zero_f32(gr->dW_hh, 3LL * H * H, st));
    BG_CUDA(bg::fill_zero_f32(gr->db_ih, 3LL * H, st));
    BG_CUDA(bg::fill_zero_f32(gr->db_hh, 3LL * H, st));
  }
  const float* gin = dET;  // gradient arriving at E(t+1)
  const bool tcg = tc_gemm_path(dt, H);
  const int64_t TN = (int64_t)T * n;
  int* status = nullptr;
  auto* Ybf = reinterpret_cast<__nv_bfloat16*>(wsc + w.Ybf);
  auto* dgib = reinterpret_cast<__nv_bfloat16*>(wsc + w.dgib);
  auto* dghb = reinterpret_cast<__nv_bfloat16*>(wsc + w.dghb);
  auto* dgiT = reinterpret_cast<__nv_bfloat16*>(wsc + w.dgiT);
  auto* dghT = reinterpret_cast<__nv_bfloat16*>(wsc + w.dghT);
  auto* YTa = reinterpret_cast<__nv_bfloat16*>(wsc + w.YTa);
  auto* ETa = reinterpret_cast<__nv_bfloat16*>(wsc + w.ETa);
  auto* WihT = reinterpret_cast<__nv_bfloat16*>(wsc + w.WihT);
  auto* WhhT = reinterpret_cast<__nv_bfloat16*>(wsc + w.WhhT);
  if (tcg) {
    BG_TRY(status_word_ptr(&status));
    // B operands W^T [H][3H] of dX = dgi W_ih and g += dgh W_hh
    BG_CUDA(bg::prep_transpose_bf16(prm->W_ih, 0, WihT, 3 * H, H, 1, st));
    BG_CUDA(bg::prep_transpose_bf16(prm->W_hh, 0, WhhT, 3 * H, H, 1, st));
  }
  for (int t = T - 1; t >= 0; --t) {
    const void* Et = sv + saved_E_off(p, dt, H, t);
    const float* Yt = reinterpret_cast<const float*>(sv + saved_Y_off(p, dt, H, T, t));
    if (tcg) {
      KTimer tm(BG_KID_GRU_BWD, st);
      BG_TRY(gru_gates_in(p, bf, H, Yt, Et, prm, gi, gh, part, pf, st, Ybf));
      BG_CUDA(bg::gru_bwd_gates(bf, gi, gh, Et, gin, dgi, dgh, g, p->n_real, n, H, st));
      BG_CUDA(bg::f32_to_bf16(dgi, dgib, (int64_t)n * 3 * H, st));
      BG_CUDA(bg::f32_to_bf16(dgh, dghb, (int64_t)n * 3 * H, st));
      BG_CUDA(bg::gemm_bf16_tn(dgib, 3 * H, 0, WihT, 3 * H, 0, n, H, 3 * H, 1, dX, H, 0, nullptr,
                               0, 0, status, st));
      BG_CUDA(bg::gemm_bf16_tn(dghb, 3 * H, 0, WhhT, 3 * H, 0, n, H, 3 * H, 1, g, H, 0, nullptr,
                               0, 1, status, st));
      // step t's columns of the weight-gradient operands (reduced after the loop)
      BG_CUDA(bg::prep_transpose_bf16(dgib, 0, dgiT + (size_t)t * n, n, 3 * H, 1, st, TN));
      BG_CUDA(bg::prep_transpose_bf16(dghb, 0, dghT + (size_t)t * n, n, 3 * H, 1, st, TN));
      BG_CUDA(bg::prep_transpose_bf16(Yt, 1, YTa + (size_t)t * n, n, H, 1, st, TN));
      BG_CUDA(bg::prep_transpose_bf16(Et, 0, ETa + (size_t)t * n, n, H, 1, st, TN));
    } else {
      KTimer tm(BG_KID_GRU_BWD, st);
      BG_TRY(gru_gates_in(p, bf, H, Yt, Et, prm, gi, gh, part, pf, st));
      // g <- direct term z * dE(t+1); dgi, dgh gate gradients
      BG_CUDA(bg::gru_bwd_gates(bf, gi, gh, Et, gin, dgi, dgh, g, p->n_real, n, H, st));
      // dX = dgi W_ih ; g += dgh W_hh
      bg::Gemm a;
      a.M = n; a.N = H; a.K = 3 * H;
      a.A = dgi; a.sAm = 3 * H; a.sAk = 1;
      a.B = prm->W_ih; a.b_bf16 = bf; a.sBk = H; a.sBn = 1;
      a.C = dX; a.ldc = H;
      BG_CUDA(bg::gemm(a, part, pf, st));
      bg::Gemm c = a;
      c.A = dgh; c.B = prm->W_hh; c.C = g; c.accumulate = 1;
      BG_CUDA(bg::gemm(c, part, pf, st));
      // dW_ih += dgi^T X ; dW_hh += dgh^T Hs ; biases
      bg::Gemm d;
      d.M = 3 * H; d.N = H; d.K = n;
      d.A = dgi; d.sAm = 1; d.sAk = 3 * H;
      d.B = Yt; d.sBk = H; d.sBn = 1;
      d.C = gr->dW_ih; d.ldc = H; d.accumulate = 1;
      BG_CUDA(bg::gemm(d, part, pf, st));
      bg::Gemm e = d;
      e.A = dgh; e.B = Et; e.b_bf16 = bf; e.C = gr->dW_hh;
      BG_CUDA(bg::gemm(e, part, pf, st));
      BG_CUDA(bg::colsum(dgi, n, 3 * H, gr->db_ih, 1, part, pf, st));
      BG_CUDA(bg::colsum(dgh, n, 3 * H, gr->db_hh, 1, part, pf, st));
    }
    // g += A^T-band backward of the messages; parameter gradients accumulate
    BG_TRY(propagate_bwd_impl(p, dt, H, Et, prm->W, dX, g, gr->dW, gr->db, 1, wsc + w.prop,
                              w.total - w.prop, st));
    if (t > 0) {
      // next iteration reads gin while writing g: keep them distinct
      BG_CUDA(cudaMemcpyAsync(dX, g, sizeof(float) * (size_t)n * H, cudaMemcpyDeviceToDevice, st));
      gin = dX;
    }
  }
  if (tcg) {
    // dW_ih, db_ih += dgi^T [Y 1] and dW_hh, db_hh += dgh^T [E 1] over all T steps at once (the
    // GEMM appends the ones column)
    KTimer tm(BG_KID_DW, st);
    const bg::TNProblem probs[2] = {
        {dgiT, TN, YTa, TN, 3 * H, 0, gr->dW_ih, gr->db_ih},
        {dghT, TN, ETa, TN, 3 * H, 0, gr->dW_hh, gr->db_hh}};
    BG_CUDA(bg::gemm_tn_multi(probs, 2, H, TN, 1, reinterpret_cast<float*>(wsc + w.tpart),
                              gru_tpart_floats(p, H, T), status, st));
  }
  BG_CUDA(cudaMemcpyAsync(dE0, g, sizeof(float) * (size_t)n * H, cudaMemcpyDeviceToDevice, st));
  return BG_OK;
}

// ---------------------------------------------------------------------------------- readout, Adam
extern "C" int bg_readout_loss(const bg_plan* p, bg_dtype dt, int32_t H, const void* ET,
                               const float* w_out, const float* target, float* loss, float* dET,
                               float* dw_out, void* ws, size_t ws_bytes, void* stream) {
  bg_clear_error();
  BG_TRY(check_plan_dev(p));
  BG_TRY(check_shape(p, dt, H));
  BG_PTR(ET, "ET"); BG_PTR(w_out, "w_out"); BG_PTR(target, "target"); BG_PTR(loss, "loss");
  BG_PTR(dET, "dET"); BG_PTR(dw_out, "dw_out"); BG_PTR(ws, "ws");
  if (ws_bytes < bg_workspace_bytes(p, dt, H, BG_OP_READOUT)) return bg_fail(BG_ECAPACITY, "workspace too small");
  float* pool = static_cast<float*>(ws);
  float* resid = pool + (size_t)p->n_packed * H;
  float* part = reinterpret_cast<float*>(static_cast<char*>(ws) +
                                         al(sizeof(float) * ((size_t)p->n_packed * H + p->n_packed + 64)));
  BG_CUDA(bg::readout_loss(dt == BG_BF16, ET, w_out, target, p->d_seg_off, p->d_seg_cnt,
                           p->d_row_graph, p->n_packed, p->n_pad(), H, pool, resid, part, loss,
                           dET, dw_out, (cudaStream_t)stream));
  return BG_OK;
}

extern "C" int bg_adam_step(int64_t n, float* master, void* working, bg_dtype wdt, float* m,
                            float* v, const float* grad, float lr, float beta1, float beta2,
                            float eps, int32_t step, void* stream) {
  bg_clear_error();
  if (n < 0) return bg_fail(BG_EINVAL, "n < 0");
  if (step < 1) return bg_fail(BG_EINVAL, "step must be >= 1");
  if (wdt != BG_F32 && wdt != BG_BF16) return bg_fail(BG_EINVAL, "unknown dtype");
  if (n == 0) return BG_OK;
  BG_PTR(master, "master"); BG_PTR(m, "m"); BG_PTR(v, "v"); BG_PTR(grad, "grad");
  BG_OPT_PTR(working, "working");
  BG_CUDA(bg::adam(n, master, working, wdt == BG_BF16, m, v, grad, lr, beta1, beta2, eps, step,
                   (cudaStream_t)stream));
  return BG_OK;
}

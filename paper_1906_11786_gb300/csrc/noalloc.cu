// bg_band_propagate_fwd_noalloc: forward band propagation whose scratch lives in a fixed,
// file-scope device array instead of a caller-provided workspace.
//
// Who needs it: code that must not allocate device memory while it runs -- for example a host
// that drives the GPU from a context where cudaMalloc is forbidden or too slow (a real-time loop,
// a memory-capped embedding in another framework's allocator, code that has pre-reserved all
// device memory), or a caller that has no allocator of its own to create the workspace tensor.
// Every other entry point takes its scratch from the caller; this one takes it from
// g_noalloc_scratch, which is part of the library image: every GPU that loads this module holds
// these kNoAllocScratchBytes until the process exits.
//
// Everything the call needs on a device is set up by bg_plan_upload (which allocates anyway):
// the array's device address, the library's status word and the forward kernels, which CUDA
// otherwise loads lazily at their first launch.  The call itself then allocates nothing.
#include <cuda_runtime.h>

#include <mutex>
#include <string>

#include "band_tc.h"
#include "internal.h"
#include "kernels.h"
#include "super.h"

namespace {

constexpr size_t kNoAllocScratchBytes = 32u << 20;  // 32 MiB

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_mu;
char* g_scratch[64] = {nullptr};

// Host code cannot use the array's name as a device address: resolve it once per device, with
// that device current.  The first resolution loads this module on the device (and reserves the
// array there).
int resolve_scratch(int dev, char** out) {
  if (dev < 0 || dev >= 64) return bg_fail(BG_EINVAL, "device index out of range");
  std::lock_guard<std::mutex> g(g_mu);
  if (!g_scratch[dev]) {
    void* s = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&s, g_noalloc_scratch);
    if (e != cudaSuccess)
      return bg_fail(BG_ECUDA, std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(e));
    g_scratch[dev] = static_cast<char*>(s);
  }
  *out = g_scratch[dev];
  return BG_OK;
}

inline size_t al(size_t x) { return (x + 255) & ~(size_t)255; }

// Scratch this entry point uses for (plan, dtype, H): the tensor-core kernels' operands (E^T, the
// second-product weights, the bias split and the split-tile partials), or the SIMT path's
// messages M_p = E W_p + b_p for every type.
size_t need_bytes(const bg_plan* p, bg_dtype dt, int H) {
  if (bg::band_tc_supported(p, (int)dt, H)) return bg::band_tc_fwd_ws_bytes(p, (int)dt, H);
  return al(sizeof(float) * (size_t)p->P * p->n_pad() * H);
}

}  // namespace

int bg_noalloc_prepare(const bg_plan* p) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return bg_fail(BG_ECUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  char* s = nullptr;
  int rc = resolve_scratch(dev, &s);
  if (rc != BG_OK) return rc;
  e = bg::preload_fwd_simt();
  if (e == cudaSuccess && p->d_maskI) e = bg::band_tc_preload_fwd(p);
  if (e == cudaSuccess) e = bg::super_preload_fwd();
  if (e != cudaSuccess) return bg_fail(BG_ECUDA, std::string("kernel load: ") + cudaGetErrorString(e));
  return BG_OK;
}

extern "C" int bg_band_propagate_fwd_noalloc(const bg_plan* p, bg_dtype dt, int32_t H,
                                             const void* E, const void* W, const float* b,
                                             float* Y, void* stream) {
  bg_clear_error();
  if (!p) return bg_fail(BG_EINVAL, "NULL plan");
  if (p->device < 0 || !p->d_masks) return bg_fail(BG_ESTATE, "plan not uploaded");
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev != p->device)
    return bg_fail(BG_ESTATE, "plan was uploaded to another device");
  if (dt != BG_F32 && dt != BG_BF16) return bg_fail(BG_EINVAL, "unknown dtype");
  if (H < 32 || H > 256 || H % 32) return bg_fail(BG_EINVAL, "H must be a multiple of 32 in [32, 256]");
  for (const void* q : {E, W, static_cast<const void*>(Y)})
    if (!q || (reinterpret_cast<uintptr_t>(q) & 15u))
      return bg_fail(BG_EINVAL, "E, W and Y must be non-NULL and 16-byte aligned");
  if (b && (reinterpret_cast<uintptr_t>(b) & 15u)) return bg_fail(BG_EINVAL, "b not 16-byte aligned");
  const size_t need = need_bytes(p, dt, H);
  if (need > kNoAllocScratchBytes)
    return bg_fail(BG_ECAPACITY, "this plan needs " + std::to_string(need) +
                                     " bytes of scratch; the static buffer of the no-allocation "
                                     "entry point holds " +
                                     std::to_string(kNoAllocScratchBytes));
  // both were set up by bg_plan_upload on this device; neither lookup allocates
  char* scratch = nullptr;
  int* status = bg_status_word_if_created(dev);
  {
    std::lock_guard<std::mutex> g(g_mu);
    scratch = g_scratch[dev];
  }
  if (!scratch || !status)
    return bg_fail(BG_ESTATE, "device not set up for the no-allocation entry point (upload the plan on it)");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (bg::band_tc_supported(p, (int)dt, H)) {
    // every byte of scratch the tensor-core path reads is written first in the same call
    e = bg::band_tc_fwd(p, H, E, W, b, Y, scratch, kNoAllocScratchBytes, status, st);
  } else {
    // SIMT path: messages M_p = E W_p + b_p into the scratch, then the band sum over the tiles
    const size_t n = (size_t)p->n_pad();
    const int bf = dt == BG_BF16;
    bg::Gemm g;
    g.M = (int)n; g.N = H; g.K = H; g.batch = p->P;
    g.A = E; g.a_bf16 = bf; g.sAb = 0; g.sAm = H; g.sAk = 1;
    g.B = W; g.b_bf16 = bf; g.sBb = (int64_t)H * H; g.sBk = H; g.sBn = 1;
    g.C = reinterpret_cast<float*>(scratch); g.sCb = (int64_t)n * H; g.ldc = H;
    g.bias = b; g.sBias = H;
    e = bg::gemm(g, nullptr, 0, st);
    if (e == cudaSuccess)
      e = bg::band_fwd_gather(p->d_masks, reinterpret_cast<float*>(scratch), Y, p->K, p->S, p->P,
                              H, st);
  }
  // the supernode rows and columns (no scratch: added to Y in place)
  if (e == cudaSuccess) e = bg::super_fwd(p, dt == BG_BF16, H, E, W, b, Y, 0, st);
  if (e != cudaSuccess) return bg_fail(BG_ECUDA, std::string("launch: ") + cudaGetErrorString(e));
  return BG_OK;
}

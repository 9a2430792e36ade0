// bg_band_propagate_fwd_noalloc: forward band propagation whose scratch lives in a fixed,
// file-scope device array instead of a caller-provided workspace.
//
// Who needs it: code that must not allocate device memory while it runs -- for example a host
// that drives the GPU from a context where cudaMalloc is forbidden or too slow (a real-time loop,
// a memory-capped embedding in another framework's allocator, code that has pre-reserved all
// device memory), or a caller that has no allocator of its own to create the workspace tensor.
// Every other entry point takes its scratch from the caller; this one takes it from
// g_noalloc_scratch, which is part of the library image: every GPU that loads the library holds
// these kNoAllocScratchBytes until the process exits.
#include <cuda_runtime.h>

#include <mutex>
#include <string>

#include "band_tc.h"
#include "internal.h"
#include "kernels.h"

namespace {

constexpr size_t kNoAllocScratchBytes = 32u << 20;  // 32 MiB

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];
// status words of the tensor-core kernels' bounded waits for calls made through this entry point
static __device__ __align__(256) int g_noalloc_status[64];

struct DevicePtrs {
  char* scratch = nullptr;
  int* status = nullptr;
};

std::mutex g_mu;
DevicePtrs g_ptrs[64];

// Host code cannot use the array's name as a device address: resolve it once per device, with
// that device current.
int device_ptrs(DevicePtrs* out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return bg_fail(BG_ECUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= 64) return bg_fail(BG_EINVAL, "device index out of range");
  std::lock_guard<std::mutex> g(g_mu);
  DevicePtrs& d = g_ptrs[dev];
  if (!d.scratch) {
    void* s = nullptr;
    void* w = nullptr;
    e = cudaGetSymbolAddress(&s, g_noalloc_scratch);
    if (e != cudaSuccess)
      return bg_fail(BG_ECUDA, std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(e));
    e = cudaGetSymbolAddress(&w, g_noalloc_status);
    if (e != cudaSuccess)
      return bg_fail(BG_ECUDA, std::string("cudaGetSymbolAddress(status): ") + cudaGetErrorString(e));
    d.scratch = static_cast<char*>(s);
    d.status = static_cast<int*>(w);
  }
  *out = d;
  return BG_OK;
}

}  // namespace

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
  const size_t need = bg_workspace_bytes(p, dt, H, BG_OP_PROPAGATE_FWD);
  if (need > kNoAllocScratchBytes)
    return bg_fail(BG_ECAPACITY, "this plan needs " + std::to_string(need) +
                                     " bytes of scratch; the static buffer of the no-allocation "
                                     "entry point holds " +
                                     std::to_string(kNoAllocScratchBytes));
  DevicePtrs d;
  int rc = device_ptrs(&d);
  if (rc != BG_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (bg::band_tc_supported(p, (int)dt, H)) {
    // every byte of scratch the tensor-core path reads is written first in the same call
    e = bg::band_tc_fwd(p, H, E, W, b, Y, d.scratch, kNoAllocScratchBytes, d.status, st);
  } else {
    // SIMT path: messages M_p = E W_p + b_p into the scratch, then the band sum over the tiles
    const size_t n = (size_t)p->n_pad();
    const int bf = dt == BG_BF16;
    bg::Gemm g;
    g.M = (int)n; g.N = H; g.K = H; g.batch = p->P;
    g.A = E; g.a_bf16 = bf; g.sAb = 0; g.sAm = H; g.sAk = 1;
    g.B = W; g.b_bf16 = bf; g.sBb = (int64_t)H * H; g.sBk = H; g.sBn = 1;
    g.C = reinterpret_cast<float*>(d.scratch); g.sCb = (int64_t)n * H; g.ldc = H;
    g.bias = b; g.sBias = H;
    e = bg::gemm(g, nullptr, 0, st);
    if (e == cudaSuccess)
      e = bg::band_fwd_gather(p->d_masks, reinterpret_cast<float*>(d.scratch), Y, p->K, p->S,
                              p->P, H, st);
  }
  if (e != cudaSuccess) return bg_fail(BG_ECUDA, std::string("launch: ") + cudaGetErrorString(e));
  return BG_OK;
}

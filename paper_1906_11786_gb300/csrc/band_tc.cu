#include "band_tc.h"

namespace bg {
bool band_tc_supported(const bg_plan*, int, int) { return false; }
size_t band_tc_fwd_ws_bytes(const bg_plan*, int, int) { return 0; }
size_t band_tc_bwd_ws_bytes(const bg_plan*, int, int) { return 0; }
cudaError_t band_tc_fwd(const bg_plan*, int, const void*, const void*, const float*, float*, char*,
                        size_t, int*, cudaStream_t) {
  return cudaErrorNotSupported;
}
cudaError_t band_tc_bwd(const bg_plan*, int, const void*, const void*, const float*, float*,
                        float*, float*, int, char*, size_t, int*, cudaStream_t) {
  return cudaErrorNotSupported;
}
void band_tc_release(bg_plan*) {}
}  // namespace bg

// sf_static.cu - sf_label_windows_noalloc: the labeler without a caller
// workspace.  Its intermediates (per-rank window medians, evidence sums, step
// leaders) live in one file-scope device array of SF_STATIC_SCRATCH_BYTES that
// every GPU loading the library holds until process exit.  The entry point
// allocates nothing: it resolves the array's device address once per device
// and hands it to sf_label_windows as the workspace.
#include <mutex>

#include "sf_launch.h"
#include "stagefrontier.h"

namespace sf {
namespace {

static __device__ __align__(256) unsigned char g_label_scratch[SF_STATIC_SCRATCH_BYTES];

constexpr int kMaxScratchDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxScratchDevices] = {};

// Device address of g_label_scratch on the current device.  In host code the
// array's name only stands in for the symbol; the address must come from the
// runtime with this device current.
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxScratchDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_label_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

}  // namespace
}  // namespace sf

extern "C" sf_status sf_label_windows_noalloc(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W,
                                              const int32_t* role, const int32_t* missing,
                                              const int64_t* wall, int32_t other_stage,
                                              const sf_label_config* cfg, uint32_t* labels,
                                              uint32_t* route_mask, uint32_t* amb_mask, double* share,
                                              double* gain, int64_t* X, int64_t* Y, int64_t* D,
                                              uint32_t* status, cudaStream_t stream) {
  const size_t need = sf_label_windows_workspace_size(T, R, S, W);
  if (need > SF_STATIC_SCRATCH_BYTES) return SF_EWORKSPACE;  // problem larger than the static scratch
  void* scratch = nullptr;
  if (need > 0 && sf::scratch_address(&scratch) != cudaSuccess) return SF_ECUDA;
  // need == 0 means invalid shape arguments: sf_label_windows reports them.
  return sf_label_windows(d, T, R, S, W, role, missing, wall, other_stage, cfg, scratch,
                          SF_STATIC_SCRATCH_BYTES, labels, route_mask, amb_mask, share, gain, X, Y, D,
                          status, stream);
}

// sf_ingest.cu - rank-major ingest.  The window-boundary gather of Sec. 5
// delivers each window as one [R][n][S] block (every rank's [n, S] buffer in
// rank order); the kernels of this library read steps as [T][R][S].  The
// conversion is a pure copy: each thread moves 16 bytes (8 when S is odd)
// of one destination row, so a warp writes 512 contiguous bytes while its
// reads are whole S*8-byte stage vectors of consecutive ranks.
#include <algorithm>
#include <cstdint>

#include "sf_device.cuh"
#include "sf_launch.h"

namespace sf {
namespace {

constexpr int kIngThreads = 256;

// dst[t][r][s] = src block b = t / N, [r][t - b*N][s]; block b starts at
// element b*R*N*S and holds n_b = min(N, T - b*N) steps.  A CTA fills one
// destination step at a time.
template <int kUnit>  // int64 values moved per thread: 2 (S even) or 1
__global__ void __launch_bounds__(kIngThreads) gathered_to_steps_kernel(const int64_t* __restrict__ src, int64_t T,
                                                                        int64_t R, int64_t S, int64_t N,
                                                                        int64_t* __restrict__ dst) {
  const int units = static_cast<int>(R * S / kUnit);  // per destination step (<= 2^21)
  const int su = static_cast<int>(S / kUnit);
  for (int64_t t = blockIdx.x; t < T; t += gridDim.x) {
    const int64_t b = t / N, tl = t - b * N;
    const int64_t nb = T - b * N < N ? T - b * N : N;
    const int64_t* sb = src + b * R * N * S + tl * S;
    int64_t* dt = dst + t * R * S;
    for (int j = threadIdx.x; j < units; j += kIngThreads) {
      const int r = j / su;
      const int s = (j - r * su) * kUnit;
      const int64_t* from = sb + int64_t(r) * nb * S + s;
      if constexpr (kUnit == 2)
        *reinterpret_cast<longlong2*>(dt + 2 * int64_t(j)) = __ldg(reinterpret_cast<const longlong2*>(from));
      else
        dt[j] = __ldg(from);
    }
  }
}

}  // namespace

cudaError_t launch_gathered_to_steps(const int64_t* src, int64_t T, int64_t R, int64_t S, int64_t N, int64_t* dst,
                                     cudaStream_t stream) {
  const int unit = S % 2 == 0 ? 2 : 1;
  const int grid = static_cast<int>(std::min<int64_t>(T, int64_t(sm_count()) * 8));
  count_launch();
  if (unit == 2)
    gathered_to_steps_kernel<2><<<grid, kIngThreads, 0, stream>>>(src, T, R, S, N, dst);
  else
    gathered_to_steps_kernel<1><<<grid, kIngThreads, 0, stream>>>(src, T, R, S, N, dst);
  return cudaGetLastError();
}

}  // namespace sf

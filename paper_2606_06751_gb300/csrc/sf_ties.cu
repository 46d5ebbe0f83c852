// sf_ties.cu - size of the lead rank's tie set per step and stage (Sec. 4:
// among the localization evidence the labeler reports the latest-rank tie
// set): ties[t,s] = #{r : P[t,r,s] = F[t,s]}, the ranks whose prefix reaches
// the frontier.  1 means the lead rank is the unique one; more means a tie
// that the frontier pass resolved to the lowest rank.
//
// One more pass over d: one CTA per step range; per step, the frontier
// F[t,s] is rebuilt from the increments a[t,.] of the frontier pass (their
// prefix over s), every thread counts, per stage, its rank rows whose prefix
// equals it, and the counts are summed over the CTA.  The per-stage state is
// sized by a bound SMAX >= S with every stage loop unrolled to SMAX behind an
// `s < S` test, so it stays in registers.
#include <algorithm>
#include <type_traits>

#include "sf_device.cuh"
#include "sf_launch.h"

namespace sf {

namespace {

constexpr int kTieThreads = 256;
constexpr int kTieWarps = kTieThreads / 32;

__device__ __forceinline__ uint32_t hi32(int64_t v) {
  return static_cast<uint32_t>(static_cast<uint64_t>(v) >> 32);
}

// VEC: S even, rows start 16-byte aligned and are read with 16-byte loads.
template <int SMAX, bool VEC>
__global__ void __launch_bounds__(kTieThreads)
    ties_kernel(const int64_t* __restrict__ d, int64_t T, int64_t R, int S, const int64_t* __restrict__ a,
                int32_t* __restrict__ ties, uint32_t* status) {
  __shared__ int64_t sF[32];
  __shared__ uint32_t wcnt[kTieWarps][32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t NB = gridDim.x, b = blockIdx.x;
  const int64_t t_begin = T * b / NB, t_end = T * (b + 1) / NB;
  uint32_t dor = 0, tor = 0;
  for (int64_t t = t_begin; t < t_end; ++t) {
    if (warp == 0) {  // F[t,s]: inclusive prefix of the increments over s
      int64_t x = lane < S ? __ldg(a + t * S + lane) : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int64_t up = __shfl_up_sync(kFull, x, o);
        if (lane >= o) x += up;
      }
      if (lane < S) sF[lane] = x;
    }
    __syncthreads();
    int64_t F[SMAX];
    uint32_t cnt[SMAX];
#pragma unroll
    for (int s = 0; s < SMAX; ++s) {
      if (s >= S) break;
      F[s] = sF[s];
      cnt[s] = 0;
    }
    for (int64_t r = threadIdx.x; r < R; r += kTieThreads) {
      const int64_t* row = d + (t * R + r) * S;
      int64_t P = 0;
      if constexpr (VEC) {
#pragma unroll
        for (int s = 0; s < SMAX; s += 2) {
          if (s >= S) break;
          const longlong2 x = __ldg(reinterpret_cast<const longlong2*>(row + s));
          dor |= hi32(x.x) | hi32(x.y);
          P += x.x;
          cnt[s] += P == F[s] ? 1u : 0u;
          P += x.y;
          cnt[s + 1] += P == F[s + 1] ? 1u : 0u;
        }
      } else {
#pragma unroll
        for (int s = 0; s < SMAX; ++s) {
          if (s >= S) break;
          const int64_t v = __ldg(row + s);
          dor |= hi32(v);
          P += v;
          cnt[s] += P == F[s] ? 1u : 0u;
        }
      }
      tor |= hi32(P);
    }
#pragma unroll
    for (int s = 0; s < SMAX; ++s) {
      if (s >= S) break;
      const uint32_t c = __reduce_add_sync(kFull, cnt[s]);
      if (lane == 0) wcnt[warp][s] = c;
    }
    __syncthreads();
    if (warp == 0 && lane < S) {
      uint32_t c = 0;
#pragma unroll
      for (int w = 0; w < kTieWarps; ++w) c += wcnt[w][lane];
      ties[t * S + lane] = static_cast<int32_t>(c);
    }
    __syncthreads();  // sF and wcnt are rewritten for the next step
  }
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), __reduce_or_sync(kFull, tor));
  if (lane == 0) report(status, bits);
}

}  // namespace

cudaError_t launch_frontier_ties(const int64_t* d, int64_t T, int64_t R, int64_t S, const int64_t* a,
                                 int32_t* ties, uint32_t* status, cudaStream_t stream) {
  const int grid = static_cast<int>(std::min<int64_t>(int64_t(sm_count()) * 4, T));
  const bool vec = S % 2 == 0;
  const int s = static_cast<int>(S);
  auto go = [&](auto smax) {
    constexpr int SM = decltype(smax)::value;
    count_launch();
    if (vec) ties_kernel<SM, true><<<grid, kTieThreads, 0, stream>>>(d, T, R, s, a, ties, status);
    else ties_kernel<SM, false><<<grid, kTieThreads, 0, stream>>>(d, T, R, s, a, ties, status);
    return cudaGetLastError();
  };
  if (S <= 4) return go(std::integral_constant<int, 4>{});
  if (S <= 8) return go(std::integral_constant<int, 8>{});
  if (S <= 16) return go(std::integral_constant<int, 16>{});
  return go(std::integral_constant<int, 32>{});
}

}  // namespace sf

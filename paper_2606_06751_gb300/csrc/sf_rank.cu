// sf_rank.cu - cross-rank order statistics per (step, stage): the lower
// median over ranks of the prefixes P[t,r,s] (for the lag of Sec. 4) or of the
// durations d[t,r,s] (for the raw rank spread of the Sec. 6 routing table),
// together with the maximum and the second largest value.
//
// One CTA per step (each CTA walks a contiguous range of steps).  A first
// pass over the step's rank rows gives every stage column its minimum, maximum
// and second largest value; then byte-digit radix passes, most significant
// first, build one 256-bin shared-memory histogram per column of the offsets
// from the column minimum (only values whose higher bytes match the digits
// chosen so far are counted) and a warp per column finds the bin holding the
// median's rank.  Each pass re-reads the step's rows, which stay in L2 (a
// step is at most R*S*8 bytes and a few hundred CTAs are in flight).
#include <algorithm>
#include <cstdint>

#include "sf_device.cuh"
#include "sf_launch.h"

namespace sf {
namespace {

constexpr int kRkThreads = 256;
constexpr int kRkWarps = kRkThreads / 32;
constexpr int kRkMaxS = 32;

struct RankParams {
  const int64_t* d;
  int64_t T, R, S;
  int of_prefix;  // 1: order statistics of P (lag); 0: of d (spread)
  int64_t t0, W, w_first;
  int64_t *L, *dL, *G;  // [T][S], nullable
  int64_t* spread;      // [nW][S], nullable
  uint32_t* status;
};

// top-2 merge: (a1 >= a2) with (b1 >= b2); a tie at the top counts as the second
__device__ __forceinline__ void top2_merge(int64_t& a1, int64_t& a2, int64_t b1, int64_t b2) {
  const int64_t n1 = a1 > b1 ? a1 : b1;
  const int64_t lo1 = a1 > b1 ? b1 : a1;
  const int64_t m2 = a2 > b2 ? a2 : b2;
  a2 = lo1 > m2 ? lo1 : m2;
  a1 = n1;
}

// SC > 0: the stage count is a compile-time constant (per-thread column state
// in registers); SC == 0: any S up to kRkMaxS.
template <int SC>
__global__ void __launch_bounds__(kRkThreads) rank_select_kernel(const RankParams p) {
  constexpr int kCols = SC > 0 ? SC : kRkMaxS;
  __shared__ __align__(16) uint32_t hist[kRkMaxS][256];
  __shared__ int64_t wmin[kRkWarps][kRkMaxS], wmax[kRkWarps][kRkMaxS], wsec[kRkWarps][kRkMaxS];
  __shared__ int64_t col_lo[kRkMaxS], col_F[kRkMaxS], col_sec[kRkMaxS];
  __shared__ uint64_t col_prefix[kRkMaxS];
  __shared__ uint32_t col_rem[kRkMaxS];
  __shared__ int col_bytes[kRkMaxS];
  __shared__ int max_bytes;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = SC > 0 ? SC : static_cast<int>(p.S);
  const int64_t R = p.R;
  const int64_t G = gridDim.x, b = blockIdx.x;
  const int64_t t_begin = p.T * b / G, t_end = p.T * (b + 1) / G;
  uint32_t dor = 0, tor = 0;
  int64_t cur_w = -1, acc = 0;  // spread accumulator of stage `lane` (warp 0)

  for (int64_t t = t_begin; t < t_end; ++t) {
    const int64_t* dt = p.d + t * R * S;
    // ---- pass 0: per-column minimum, maximum and second largest
    int64_t mn[kCols], m1[kCols], m2[kCols];
#pragma unroll
    for (int s = 0; s < kCols; ++s) {
      mn[s] = INT64_MAX;
      m1[s] = -1;
      m2[s] = -1;
    }
    for (int64_t r = threadIdx.x; r < R; r += kRkThreads) {
      int64_t P = 0;
#pragma unroll
      for (int s = 0; s < kCols; ++s) {
        if (SC == 0 && s >= S) break;
        const int64_t v = __ldg(dt + r * S + s);
        dor |= static_cast<uint32_t>(static_cast<uint64_t>(v) >> 32);
        P += v;
        const int64_t x = p.of_prefix ? P : v;
        mn[s] = x < mn[s] ? x : mn[s];
        top2_merge(m1[s], m2[s], x, -1);
      }
      tor |= static_cast<uint32_t>(static_cast<uint64_t>(P) >> 32);
    }
#pragma unroll
    for (int s = 0; s < kCols; ++s) {
      if (SC == 0 && s >= S) break;
      int64_t a = mn[s], x1 = m1[s], x2 = m2[s];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const int64_t oa = __shfl_xor_sync(kFull, a, o);
        const int64_t o1 = __shfl_xor_sync(kFull, x1, o);
        const int64_t o2 = __shfl_xor_sync(kFull, x2, o);
        a = oa < a ? oa : a;
        top2_merge(x1, x2, o1, o2);
      }
      if (lane == 0) {
        wmin[warp][s] = a;
        wmax[warp][s] = x1;
        wsec[warp][s] = x2;
      }
    }
    __syncthreads();
    if (threadIdx.x < S) {
      const int s = threadIdx.x;
      int64_t a = wmin[0][s], x1 = wmax[0][s], x2 = wsec[0][s];
      for (int w = 1; w < kRkWarps; ++w) {
        a = wmin[w][s] < a ? wmin[w][s] : a;
        top2_merge(x1, x2, wmax[w][s], wsec[w][s]);
      }
      col_lo[s] = a;
      col_F[s] = x1;
      col_sec[s] = R >= 2 ? x2 : x1;
      const uint64_t range = static_cast<uint64_t>(x1 - a);
      col_bytes[s] = range ? (64 - __clzll(static_cast<long long>(range)) + 7) / 8 : 0;
      col_prefix[s] = 0;
      col_rem[s] = static_cast<uint32_t>((R - 1) / 2);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int mb = 0;
      for (int s = 0; s < S; ++s) mb = col_bytes[s] > mb ? col_bytes[s] : mb;
      max_bytes = mb;
    }
    __syncthreads();
    // ---- byte passes, most significant first
    for (int bb = max_bytes - 1; bb >= 0; --bb) {
      for (int i = threadIdx.x; i < S * 256; i += kRkThreads) hist[i >> 8][i & 255] = 0;
      __syncthreads();
      const int sh = 8 * bb;
      for (int64_t r = threadIdx.x; r < R; r += kRkThreads) {
        int64_t P = 0;
        for (int s = 0; s < S; ++s) {
          const int64_t v = __ldg(dt + r * S + s);
          P += v;
          if (bb < col_bytes[s]) {
            const uint64_t off = static_cast<uint64_t>((p.of_prefix ? P : v) - col_lo[s]);
            const bool match = sh + 8 >= 64 || (off >> (sh + 8)) == (col_prefix[s] >> (sh + 8));
            if (match) atomicAdd(&hist[s][static_cast<uint32_t>(off >> sh) & 255u], 1u);
          }
        }
      }
      __syncthreads();
      for (int s = warp; s < S; s += kRkWarps) {
        if (bb < col_bytes[s]) {
          uint32_t digit, below;
          hist_find(hist[s], col_rem[s], lane, digit, below);
          __syncwarp();
          if (lane == 0) {
            col_rem[s] -= below;
            col_prefix[s] |= static_cast<uint64_t>(digit) << sh;
          }
        }
      }
      __syncthreads();
    }
    // ---- per-step outputs
    if (warp == 0) {
      const bool valid = lane < S;
      const int64_t med = valid ? col_lo[lane] + static_cast<int64_t>(col_prefix[lane]) : 0;
      const int64_t F = valid ? col_F[lane] : 0;
      if (p.of_prefix) {
        const int64_t lag = F - med;
        int64_t prev = __shfl_up_sync(kFull, lag, 1);
        if (lane == 0) prev = 0;
        if (valid) {
          if (p.L) p.L[t * S + lane] = lag;
          if (p.dL) p.dL[t * S + lane] = lag - prev;
          if (p.G) p.G[t * S + lane] = F - col_sec[lane];
        }
      } else {
        const int64_t w = (p.t0 + t) / p.W - p.w_first;
        if (w != cur_w) {
          if (cur_w >= 0 && valid && acc)
            atomicAdd(reinterpret_cast<unsigned long long*>(&p.spread[cur_w * S + lane]),
                      static_cast<unsigned long long>(acc));
          acc = 0;
          cur_w = w;
        }
        acc += valid ? F - med : 0;
      }
    }
    __syncthreads();  // column state is rewritten by the next step
  }
  if (!p.of_prefix && warp == 0 && cur_w >= 0 && lane < S && acc)
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.spread[cur_w * S + lane]),
              static_cast<unsigned long long>(acc));
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), p.of_prefix ? __reduce_or_sync(kFull, tor) : 0u);
  if (lane == 0) report(p.status, bits);
}

}  // namespace

cudaError_t launch_rank_select(const int64_t* d, int64_t T, int64_t R, int64_t S, int of_prefix, int64_t t0,
                               int64_t W, int64_t* L, int64_t* dL, int64_t* G, int64_t* spread, uint32_t* status,
                               cudaStream_t stream) {
  RankParams p{};
  p.d = d;
  p.T = T;
  p.R = R;
  p.S = S;
  p.of_prefix = of_prefix;
  p.t0 = t0;
  p.W = W;
  p.w_first = t0 / W;
  p.L = L;
  p.dL = dL;
  p.G = G;
  p.spread = spread;
  p.status = status;
  // each CTA re-reads its current step once per byte pass: keep the steps in
  // flight within about half of L2
  const int64_t sms = sm_count();
  const int64_t fit = std::max<int64_t>(sms, (int64_t(64) << 20) / (R * S * 8));
  const int grid = static_cast<int>(std::min<int64_t>(std::min<int64_t>(sms * 4, fit), T));
  count_launch();
  switch (S) {
    case 4: rank_select_kernel<4><<<grid, kRkThreads, 0, stream>>>(p); break;
    case 6: rank_select_kernel<6><<<grid, kRkThreads, 0, stream>>>(p); break;
    case 8: rank_select_kernel<8><<<grid, kRkThreads, 0, stream>>>(p); break;
    case 10: rank_select_kernel<10><<<grid, kRkThreads, 0, stream>>>(p); break;
    case 16: rank_select_kernel<16><<<grid, kRkThreads, 0, stream>>>(p); break;
    default: rank_select_kernel<0><<<grid, kRkThreads, 0, stream>>>(p); break;
  }
  return cudaGetLastError();
}

}  // namespace sf

// sf_group.cu - the frontier taken within role groups (the App. A role check:
// no global frontier across ranks whose roles differ; Sec. 3 Eq. 1 applied
// inside each group) and reporting-group sums after the frontier (Sec. 3:
// accumulation-indexed stages are aggregated only once the frontier is taken).
//
// group_window_kernel: a CTA walks a contiguous range of steps.  For each
// step its threads stream the rank rows (16-byte loads, two rows in flight,
// the stage prefix in registers) and fold every prefix into a shared-memory
// maximum per (group, stage).  When all 32 lanes of a warp hold ranks of one
// group - the common case of contiguous node groups - the warp first reduces
// each stage in registers and issues one shared atomic; otherwise every lane
// issues its own.  The per-group increments F_g[s] - F_g[s-1] and makespans
// then accumulate in shared memory per window and are added to global memory
// once per window the CTA touches.
#include <algorithm>
#include <cstdint>

#include "sf_device.cuh"
#include "sf_launch.h"

namespace sf {
namespace {

constexpr int kGrThreads = 256;

struct GroupParams {
  const int64_t* d;
  int64_t T, R, S;
  const int32_t* group;
  int64_t G, t0, W, w_first;
  int64_t* Xg;  // [nW][G][S]
  int64_t* Dg;  // [nW][G]
  uint32_t* status;
};

__device__ __forceinline__ unsigned long long warp_max_u64_all(unsigned long long v) {
  const uint32_t hi = __reduce_max_sync(kFull, static_cast<uint32_t>(v >> 32));
  const uint32_t lo = __reduce_max_sync(kFull, static_cast<uint32_t>(v >> 32) == hi ? static_cast<uint32_t>(v) : 0u);
  return (static_cast<unsigned long long>(hi) << 32) | lo;
}

// One rank row: the stage prefix folded into the group's per-stage maximum.
template <int SC>
__device__ __forceinline__ void fold_row(const GroupParams& p, const int64_t* row, int S, int g, bool valid,
                                         bool warp_uniform, unsigned long long* Fk, uint32_t& dor, uint32_t& tor) {
  constexpr int kCols = SC > 0 ? SC : 1;
  int64_t P = 0;
  if constexpr (SC > 0) {
    int64_t v[kCols];
    if (valid) {
      if constexpr (SC % 2 == 0) {
#pragma unroll
        for (int h = 0; h < SC / 2; ++h) {
          const longlong2 x = __ldg(reinterpret_cast<const longlong2*>(row) + h);
          v[2 * h] = x.x;
          v[2 * h + 1] = x.y;
        }
      } else {
#pragma unroll
        for (int s = 0; s < SC; ++s) v[s] = __ldg(row + s);
      }
    } else {
#pragma unroll
      for (int s = 0; s < SC; ++s) v[s] = 0;
    }
#pragma unroll
    for (int s = 0; s < SC; ++s) {
      dor |= static_cast<uint32_t>(static_cast<uint64_t>(v[s]) >> 32);
      P += v[s];
      if (warp_uniform) {
        const unsigned long long m = warp_max_u64_all(static_cast<unsigned long long>(P));
        if ((threadIdx.x & 31) == 0) atomicMax(&Fk[g * SC + s], m);
      } else if (valid) {
        atomicMax(&Fk[g * SC + s], static_cast<unsigned long long>(P));
      }
    }
  } else {
    for (int s = 0; s < S; ++s) {
      const int64_t v = valid ? __ldg(row + s) : 0;
      dor |= static_cast<uint32_t>(static_cast<uint64_t>(v) >> 32);
      P += v;
      if (warp_uniform) {
        const unsigned long long m = warp_max_u64_all(static_cast<unsigned long long>(P));
        if ((threadIdx.x & 31) == 0) atomicMax(&Fk[g * S + s], m);
      } else if (valid) {
        atomicMax(&Fk[g * S + s], static_cast<unsigned long long>(P));
      }
    }
  }
  tor |= static_cast<uint32_t>(static_cast<uint64_t>(P) >> 32);
}

// Dynamic shared memory: Fk [G][S] u64 (this step's group frontier),
// accX [G][S] i64 and accD [G] i64 (the current window's sums).
template <int SC>
__global__ void __launch_bounds__(kGrThreads) group_window_kernel(const GroupParams p) {
  extern __shared__ __align__(16) unsigned char dyn[];
  const int S = SC > 0 ? SC : static_cast<int>(p.S);
  const int G = static_cast<int>(p.G), GS = G * S;
  unsigned long long* Fk = reinterpret_cast<unsigned long long*>(dyn);
  int64_t* accX = reinterpret_cast<int64_t*>(Fk + GS);
  int64_t* accD = accX + GS;
  const int tid = threadIdx.x, lane = tid & 31;
  const int64_t R = p.R;
  const int64_t nb = gridDim.x, b = blockIdx.x;
  const int64_t q = p.T / nb, rr = p.T % nb;
  const int64_t t_begin = q * b + (b < rr ? b : rr), t_end = t_begin + q + (b < rr ? 1 : 0);
  uint32_t dor = 0, tor = 0, bad_group = 0;
  int64_t cur_w = -1;
  int64_t w = 0, w_lo = 0, w_hi = 0;  // steps [w_lo, w_hi) form window w: one division per window

  for (int i = tid; i < GS + G; i += kGrThreads) accX[i] = 0;  // accX and accD are contiguous
  for (int64_t t = t_begin; t < t_end; ++t) {
    if (t < w_lo || t >= w_hi) {
      w = (p.t0 + t) / p.W - p.w_first;
      w_lo = (w + p.w_first) * p.W - p.t0;
      w_hi = w_lo + p.W;
    }
    for (int i = tid; i < GS; i += kGrThreads) Fk[i] = 0;
    if (w != cur_w && cur_w >= 0) {
      // the window changed: add the finished window's sums to global memory
      for (int i = tid; i < GS; i += kGrThreads) {
        if (accX[i]) atomicAdd(reinterpret_cast<unsigned long long*>(&p.Xg[cur_w * GS + i]),
                               static_cast<unsigned long long>(accX[i]));
        accX[i] = 0;
      }
      for (int g = tid; g < G; g += kGrThreads) {
        if (accD[g]) atomicAdd(reinterpret_cast<unsigned long long*>(&p.Dg[cur_w * G + g]),
                               static_cast<unsigned long long>(accD[g]));
        accD[g] = 0;
      }
    }
    cur_w = w;
    __syncthreads();
    const int64_t* dt = p.d + t * R * S;
    constexpr int kRows = (SC > 0 && SC <= 8) ? 2 : 1;
    for (int64_t base = tid - lane; base < R; base += int64_t(kRows) * kGrThreads) {
      // warp-uniform loop: every lane takes part in the warp reductions
#pragma unroll
      for (int k = 0; k < kRows; ++k) {
        const int64_t r = base + int64_t(k) * kGrThreads + lane;
        const bool in = r < R;
        int g = in ? __ldg(p.group + r) : -1;
        const bool ok = g >= 0 && g < G;
        bad_group |= (in && !ok) ? 1u : 0u;
        if (!ok) g = 0;
        const int g0 = __shfl_sync(kFull, g, 0);
        const bool uniform = __all_sync(kFull, ok && g == g0);
        fold_row<SC>(p, dt + (in ? r : 0) * S, S, g, ok, uniform, Fk, dor, tor);
      }
    }
    __syncthreads();
    // the step's group increments a_g[s] = F_g[s] - F_g[s-1] and makespans
    for (int i = tid; i < GS; i += kGrThreads) {
      const int s = i % S;
      const int64_t F = static_cast<int64_t>(Fk[i]);
      accX[i] += F - (s > 0 ? static_cast<int64_t>(Fk[i - 1]) : 0);
      if (s == S - 1) accD[i / S] += F;
    }
    __syncthreads();
  }
  if (cur_w >= 0) {
    for (int i = tid; i < GS; i += kGrThreads)
      if (accX[i]) atomicAdd(reinterpret_cast<unsigned long long*>(&p.Xg[cur_w * GS + i]),
                             static_cast<unsigned long long>(accX[i]));
    for (int g = tid; g < G; g += kGrThreads)
      if (accD[g]) atomicAdd(reinterpret_cast<unsigned long long*>(&p.Dg[cur_w * G + g]),
                             static_cast<unsigned long long>(accD[g]));
  }
  uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), __reduce_or_sync(kFull, tor));
  if (__any_sync(kFull, bad_group != 0)) bits |= SF_ST_INDEX;
  if (lane == 0) report(p.status, bits);
}

struct StageGroups {
  int32_t of[32];  // stage -> reporting group
};

__global__ void stage_group_sum_kernel(const int64_t* __restrict__ X, int64_t nW, int S, StageGroups sg, int K,
                                       int64_t* __restrict__ Y) {
  const int64_t n = nW * K;
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n; i += int64_t(gridDim.x) * blockDim.x) {
    const int64_t w = i / K;
    const int k = static_cast<int>(i - w * K);
    int64_t y = 0;
    for (int s = 0; s < S; ++s)
      if (sg.of[s] == k) y += X[w * S + s];
    Y[i] = y;
  }
}

template <int SC>
cudaError_t launch_group_t(const GroupParams& p, size_t smem, cudaStream_t stream) {
  auto kern = group_window_kernel<SC>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kGrThreads, smem) != cudaSuccess || per_sm < 1) {
    cudaGetLastError();
    per_sm = 1;
  }
  const int grid = static_cast<int>(std::min<int64_t>(int64_t(per_sm) * sm_count(), p.T));
  count_launch();
  kern<<<grid, kGrThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_group_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, const int32_t* group, int64_t G,
                                 int64_t t0, int64_t W, int64_t* Xg, int64_t* Dg, uint32_t* status,
                                 cudaStream_t stream) {
  GroupParams p{};
  p.d = d;
  p.T = T;
  p.R = R;
  p.S = S;
  p.group = group;
  p.G = G;
  p.t0 = t0;
  p.W = W;
  p.w_first = t0 / W;
  p.Xg = Xg;
  p.Dg = Dg;
  p.status = status;
  const size_t smem = size_t(G) * S * 16 + size_t(G) * 8;
  switch (S) {
    case 4: return launch_group_t<4>(p, smem, stream);
    case 6: return launch_group_t<6>(p, smem, stream);
    case 8: return launch_group_t<8>(p, smem, stream);
    case 10: return launch_group_t<10>(p, smem, stream);
    case 16: return launch_group_t<16>(p, smem, stream);
    default: return launch_group_t<0>(p, smem, stream);
  }
}

cudaError_t launch_stage_group_sum(const int64_t* X, int64_t nW, int64_t S, const int32_t* stage_group, int64_t K,
                                   int64_t* Y, cudaStream_t stream) {
  StageGroups sg{};
  for (int s = 0; s < S; ++s) sg.of[s] = stage_group[s];
  const int64_t n = nW * K;
  const int grid = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>((n + 255) / 256, int64_t(sm_count()) * 8)));
  count_launch();
  stage_group_sum_kernel<<<grid, 256, 0, stream>>>(X, nW, static_cast<int>(S), sg, static_cast<int>(K), Y);
  return cudaGetLastError();
}

}  // namespace sf

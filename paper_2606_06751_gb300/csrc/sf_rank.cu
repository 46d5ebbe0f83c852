// sf_rank.cu - cross-rank order statistics per (step, stage): the lower
// median over ranks of the prefixes P[t,r,s] (for the lag of Sec. 4) or of the
// durations d[t,r,s] (for the raw rank spread of the Sec. 6 routing table),
// together with the maximum and the second largest value.
//
// rank_keys_kernel - a cluster of C CTAs per step (C = 1, 2, 4 or 8: the
//   smallest whose shared memory holds the step), the CTAs splitting the
//   step's rank rows.  Each CTA reads its rows once from HBM with 16-byte
//   loads, sums the stage prefix in registers and stores every column as
//   32-bit keys: the value minus rank 0's value, sign bit flipped, so that
//   unsigned key order is value order.  A step with a value 2^31 or more away
//   from rank 0's is handed to the 64-bit path below.  One pass over the keys
//   gives each column's minimum, maximum and second largest key, merged over
//   the cluster through distributed shared memory.  Radix passes then count
//   the key offsets from the column minimum, top digit first; the top digit
//   starts at the highest bit of the column's range so that it spreads over
//   the 256 bins.  Each CTA counts its own rows into its own histogram (two
//   buffers, alternating by pass); after one cluster barrier every CTA sums
//   the cluster's histograms and finds the same digit, so the CTAs stay in
//   step without any further exchange.
// rank_global_kernel - steps too large for eight CTAs' shared memory: a CTA
//   per step re-reads the 64-bit rows from L2 once per byte of the range.
#include <cooperative_groups.h>

#include <algorithm>
#include <cstdint>

#include "sf_device.cuh"
#include "sf_launch.h"

namespace cg = cooperative_groups;

namespace sf {
namespace {

constexpr int kRkThreads = 256;
constexpr int kRkWarps = kRkThreads / 32;
constexpr int kRkMaxS = 32;
constexpr size_t kRkSmemTwoPerSm = 100 * 1024;  // dynamic shared memory that leaves room for two CTAs per SM
constexpr size_t kRkSmemOnePerSm = 200 * 1024;

struct RankParams {
  const int64_t* d;
  int64_t T, R, S;
  int of_prefix;  // 1: order statistics of P (lag); 0: of d (spread)
  int64_t t0, W, w_first;
  int64_t *L, *dL, *G;  // [T][S], nullable
  int64_t* spread;      // [nW][S], nullable
  uint32_t* status;
  int64_t Rc;  // rank rows per CTA of a cluster
  int64_t ld;  // column stride of the key slab (a multiple of 4)
};

// One step's per-column results, in the shared memory of the CTA that writes them.
struct StepOut {
  int64_t med[kRkMaxS], F[kRkMaxS], sec[kRkMaxS];
};

// top-2 merge: (a1 >= a2) with (b1 >= b2); a tie at the top counts as the second
template <typename V>
__device__ __forceinline__ void top2_merge(V& a1, V& a2, V b1, V b2) {
  const V n1 = a1 > b1 ? a1 : b1;
  const V lo1 = a1 > b1 ? b1 : a1;
  const V m2 = a2 > b2 ? a2 : b2;
  a2 = lo1 > m2 ? lo1 : m2;
  a1 = n1;
}

// [begin, end) of part b of n parts of [0, T), balanced, without overflow
__device__ __forceinline__ void split_range(int64_t T, int64_t n, int64_t b, int64_t& begin, int64_t& end) {
  const int64_t q = T / n, r = T % n;
  begin = q * b + (b < r ? b : r);
  end = begin + q + (b < r ? 1 : 0);
}

// The outputs of one step, written by warp 0 of the step's writer CTA: lag,
// delta-lag and gap per stage, or the window's spread accumulated in
// registers (lane = stage) and added to global memory when the window changes.
struct Emitter {
  int64_t cur_w = -1, acc = 0;

  __device__ __forceinline__ void step(const RankParams& p, int64_t t, const StepOut& o, int lane) {
    const int S = static_cast<int>(p.S);
    const bool valid = lane < S;
    const int64_t med = valid ? o.med[lane] : 0;
    const int64_t F = valid ? o.F[lane] : 0;
    if (p.of_prefix) {
      const int64_t lag = F - med;
      int64_t prev = __shfl_up_sync(kFull, lag, 1);
      if (lane == 0) prev = 0;
      if (valid) {
        if (p.L) p.L[t * S + lane] = lag;
        if (p.dL) p.dL[t * S + lane] = lag - prev;
        if (p.G) p.G[t * S + lane] = F - o.sec[lane];
      }
    } else {
      const int64_t w = (p.t0 + t) / p.W - p.w_first;
      if (w != cur_w) {
        flush(p, lane);
        cur_w = w;
      }
      acc += valid ? F - med : 0;
    }
  }

  __device__ __forceinline__ void flush(const RankParams& p, int lane) {
    if (!p.of_prefix && cur_w >= 0 && lane < p.S && acc)
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.spread[cur_w * p.S + lane]),
                static_cast<unsigned long long>(acc));
    acc = 0;
  }
};

// ---------------------------------------------------------------- 64-bit path

struct Global64 {
  // per-warp partials: [warp][column] in the 64-bit kernel (8 warps); [0][warp]
  // in the key kernel's out-of-range path (one column at a time, up to 32 warps)
  int64_t wmin[kRkWarps][kRkMaxS], wmax[kRkWarps][kRkMaxS], wsec[kRkWarps][kRkMaxS];
  int64_t lo[kRkMaxS];
  uint64_t prefix[kRkMaxS];
  uint32_t rem[kRkMaxS];
  int bytes[kRkMaxS];
  int max_bytes;
};

// One step by one CTA on the 64-bit values in global memory: a pass for each
// column's minimum, maximum and second largest, then one pass per byte of the
// column range (offsets from the minimum, most significant byte first), each
// counting the values that match the bytes chosen so far into hist[s][256].
// Leaves med/F/sec in `out`; ends with a CTA barrier.
template <int SC>
__device__ void select_step_global(const RankParams& p, int64_t t, uint32_t* hist, Global64& g, StepOut& out,
                                   uint32_t& dor, uint32_t& tor) {
  constexpr int kCols = SC > 0 ? SC : kRkMaxS;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = SC > 0 ? SC : static_cast<int>(p.S);
  const int64_t R = p.R;
  const int64_t* dt = p.d + t * R * S;
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
      top2_merge<int64_t>(m1[s], m2[s], x, -1);
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
      top2_merge<int64_t>(x1, x2, o1, o2);
    }
    if (lane == 0) {
      g.wmin[warp][s] = a;
      g.wmax[warp][s] = x1;
      g.wsec[warp][s] = x2;
    }
  }
  __syncthreads();
  if (threadIdx.x < S) {
    const int s = threadIdx.x;
    int64_t a = g.wmin[0][s], x1 = g.wmax[0][s], x2 = g.wsec[0][s];
    for (int w = 1; w < kRkWarps; ++w) {
      a = g.wmin[w][s] < a ? g.wmin[w][s] : a;
      top2_merge<int64_t>(x1, x2, g.wmax[w][s], g.wsec[w][s]);
    }
    g.lo[s] = a;
    out.F[s] = x1;
    out.sec[s] = R >= 2 ? x2 : x1;
    const uint64_t range = static_cast<uint64_t>(x1 - a);
    g.bytes[s] = range ? (64 - __clzll(static_cast<long long>(range)) + 7) / 8 : 0;
    g.prefix[s] = 0;
    g.rem[s] = static_cast<uint32_t>((R - 1) / 2);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int mb = 0;
    for (int s = 0; s < S; ++s) mb = g.bytes[s] > mb ? g.bytes[s] : mb;
    g.max_bytes = mb;
  }
  __syncthreads();
  for (int bb = g.max_bytes - 1; bb >= 0; --bb) {
    for (int i = threadIdx.x; i < S * 256; i += kRkThreads) hist[i] = 0;
    __syncthreads();
    const int sh = 8 * bb;
    for (int64_t r = threadIdx.x; r < R; r += kRkThreads) {
      int64_t P = 0;
      for (int s = 0; s < S; ++s) {
        const int64_t v = __ldg(dt + r * S + s);
        P += v;
        if (bb < g.bytes[s]) {
          const uint64_t off = static_cast<uint64_t>((p.of_prefix ? P : v) - g.lo[s]);
          const bool match = sh + 8 >= 64 || (off >> (sh + 8)) == (g.prefix[s] >> (sh + 8));
          if (match) atomicAdd(&hist[s * 256 + (static_cast<uint32_t>(off >> sh) & 255u)], 1u);
        }
      }
    }
    __syncthreads();
    for (int s = warp; s < S; s += kRkWarps) {
      if (bb < g.bytes[s]) {
        uint32_t digit, below;
        hist_find(hist + s * 256, g.rem[s], lane, digit, below);
        if (lane == 0) {
          g.rem[s] -= below;
          g.prefix[s] |= static_cast<uint64_t>(digit) << sh;
        }
      }
    }
    __syncthreads();
  }
  if (threadIdx.x < S) out.med[threadIdx.x] = g.lo[threadIdx.x] + static_cast<int64_t>(g.prefix[threadIdx.x]);
  __syncthreads();
}

// The 64-bit path for one step of the key kernel, one column at a time so
// that it holds no per-column registers (its prefix is re-summed from the
// row for every column); the key kernel calls it for the rare step whose
// values lie 2^31 or more from rank 0's.  The status bits were already taken
// by the key kernel's load.  Ends with a CTA barrier.
__device__ __forceinline__ void select_step_lean(const RankParams& p, int64_t t, uint32_t* hist, Global64& g,
                                              StepOut& out) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nt = blockDim.x, nw = nt >> 5;  // any CTA width up to 32 warps
  const int S = static_cast<int>(p.S);
  const int64_t R = p.R;
  const int64_t* dt = p.d + t * R * S;
  auto value = [&](int64_t r, int s) {
    const int64_t* row = dt + r * S;
    if (!p.of_prefix) return __ldg(row + s);
    int64_t P = 0;
    for (int i = 0; i <= s; ++i) P += __ldg(row + i);
    return P;
  };
  for (int s = 0; s < S; ++s) {
    int64_t a = INT64_MAX, x1 = -1, x2 = -1;
    for (int64_t r = threadIdx.x; r < R; r += nt) {
      const int64_t x = value(r, s);
      a = x < a ? x : a;
      top2_merge<int64_t>(x1, x2, x, -1);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const int64_t oa = __shfl_xor_sync(kFull, a, o);
      const int64_t o1 = __shfl_xor_sync(kFull, x1, o);
      const int64_t o2 = __shfl_xor_sync(kFull, x2, o);
      a = oa < a ? oa : a;
      top2_merge<int64_t>(x1, x2, o1, o2);
    }
    if (lane == 0) {
      g.wmin[0][warp] = a;
      g.wmax[0][warp] = x1;
      g.wsec[0][warp] = x2;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      a = g.wmin[0][0];
      x1 = g.wmax[0][0];
      x2 = g.wsec[0][0];
      for (int w = 1; w < nw; ++w) {
        a = g.wmin[0][w] < a ? g.wmin[0][w] : a;
        top2_merge<int64_t>(x1, x2, g.wmax[0][w], g.wsec[0][w]);
      }
      g.lo[0] = a;
      out.F[s] = x1;
      out.sec[s] = R >= 2 ? x2 : x1;
      const uint64_t range = static_cast<uint64_t>(x1 - a);
      g.bytes[0] = range ? (64 - __clzll(static_cast<long long>(range)) + 7) / 8 : 0;
      g.prefix[0] = 0;
      g.rem[0] = static_cast<uint32_t>((R - 1) / 2);
    }
    __syncthreads();
    for (int bb = g.bytes[0] - 1; bb >= 0; --bb) {
      for (int i = threadIdx.x; i < 256; i += nt) hist[i] = 0;
      __syncthreads();
      const int sh = 8 * bb;
      const int64_t lo = g.lo[0];
      const uint64_t pref = g.prefix[0];
      for (int64_t r = threadIdx.x; r < R; r += nt) {
        const uint64_t off = static_cast<uint64_t>(value(r, s) - lo);
        if (sh + 8 >= 64 || (off >> (sh + 8)) == (pref >> (sh + 8)))
          atomicAdd(&hist[static_cast<uint32_t>(off >> sh) & 255u], 1u);
      }
      __syncthreads();
      if (warp == 0) {
        uint32_t digit, below;
        hist_find(hist, g.rem[0], lane, digit, below);
        if (lane == 0) {
          g.rem[0] -= below;
          g.prefix[0] |= static_cast<uint64_t>(digit) << sh;
        }
      }
      __syncthreads();
    }
    if (threadIdx.x == 0) out.med[s] = g.lo[0] + static_cast<int64_t>(g.prefix[0]);
    __syncthreads();
  }
}

template <int SC>
__global__ void __launch_bounds__(kRkThreads) rank_global_kernel(const RankParams p) {
  __shared__ __align__(16) uint32_t hist[kRkMaxS * 256];
  __shared__ Global64 g;
  __shared__ StepOut out;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int64_t t_begin, t_end;
  split_range(p.T, gridDim.x, blockIdx.x, t_begin, t_end);
  uint32_t dor = 0, tor = 0;
  Emitter em;
  for (int64_t t = t_begin; t < t_end; ++t) {
    select_step_global<SC>(p, t, hist, g, out, dor, tor);
    if (warp == 0) em.step(p, t, out, lane);
    __syncthreads();  // `out` and the column state are rewritten by the next step
  }
  if (warp == 0) em.flush(p, lane);
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), p.of_prefix ? __reduce_or_sync(kFull, tor) : 0u);
  if (lane == 0) report(p.status, bits);
}

// ------------------------------------------------------------ 32-bit key path

constexpr int kKeyThreads = 384;
constexpr int kKeyWarps = kKeyThreads / 32;
constexpr int kCand = 256;  // candidate keys per column a CTA keeps after the second pass

struct KeyState {
  // this CTA's column statistics and out-of-range flag, by step parity: the
  // cluster's other CTAs read them after the step's first cluster barrier
  uint32_t cmn[2][kRkMaxS], cmx[2][kRkMaxS], csc[2][kRkMaxS];
  uint32_t cbad[2];
  uint32_t pmn[kRkMaxS], pmx[kRkMaxS], psc[kRkMaxS];  // partial statistics, one per (column, row part)
  int64_t ref[kRkMaxS];    // rank 0's value per column
  uint32_t lo[kRkMaxS];    // column minimum key (cluster-wide)
  uint32_t pref[kRkMaxS];  // offset bits chosen so far
  uint32_t rem[kRkMaxS];   // rank still sought among the matching offsets
  int nb[kRkMaxS];         // bit length of the column's key range
  uint32_t ncand[kRkMaxS];  // candidates kept for the column (third pass on)
  int compact[kRkMaxS];     // 1: the column's candidates fit in kCand and later passes read only them
  int bad;
};

__device__ __forceinline__ int64_t key_value(int64_t ref, uint32_t key) {
  return ref + static_cast<int64_t>(static_cast<int32_t>(key ^ 0x80000000u));
}

// Stage values of one rank row: P (of_prefix) or d, minus rank 0's value, as
// keys in column s of the slab at row rl.  Returns whether a value lay 2^31
// or more away from rank 0's.
template <int SC>
__device__ __forceinline__ bool store_row(const RankParams& p, const int64_t* row, int S, const KeyState& ks,
                                          uint32_t* keys, int rl, uint32_t& dor, uint32_t& tor) {
  bool bad = false;
  int64_t P = 0;
  const int ld = static_cast<int>(p.ld);
  if constexpr (SC > 0 && SC % 2 == 0) {
    int64_t v[SC];
#pragma unroll
    for (int h = 0; h < SC / 2; ++h) {
      const longlong2 x = __ldg(reinterpret_cast<const longlong2*>(row) + h);
      v[2 * h] = x.x;
      v[2 * h + 1] = x.y;
    }
#pragma unroll
    for (int s = 0; s < SC; ++s) {
      dor |= static_cast<uint32_t>(static_cast<uint64_t>(v[s]) >> 32);
      P += v[s];
      const int64_t diff = (p.of_prefix ? P : v[s]) - ks.ref[s];
      bad |= (static_cast<uint64_t>(diff + 0x80000000ll) >> 32) != 0;
      keys[s * ld + rl] = static_cast<uint32_t>(diff) ^ 0x80000000u;
    }
  } else {
    for (int s = 0; s < S; ++s) {
      const int64_t v = __ldg(row + s);
      dor |= static_cast<uint32_t>(static_cast<uint64_t>(v) >> 32);
      P += v;
      const int64_t diff = (p.of_prefix ? P : v) - ks.ref[s];
      bad |= (static_cast<uint64_t>(diff + 0x80000000ll) >> 32) != 0;
      keys[s * ld + rl] = static_cast<uint32_t>(diff) ^ 0x80000000u;
    }
  }
  tor |= static_cast<uint32_t>(static_cast<uint64_t>(P) >> 32);
  return bad;
}

// Dynamic shared memory: hist [2][S][256] u32, cand [S][kCand] u32, keys [S][ld] u32.
template <int SC>
__global__ void __launch_bounds__(kKeyThreads, 2) rank_keys_kernel(const RankParams p) {
  extern __shared__ __align__(16) unsigned char dyn[];
  __shared__ KeyState ks;
  __shared__ Global64 g;
  __shared__ StepOut out;
  cg::cluster_group cluster = cg::this_cluster();
  const unsigned C = cluster.num_blocks(), q = cluster.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int S = SC > 0 ? SC : static_cast<int>(p.S);
  const int64_t R = p.R;
  const int ld = static_cast<int>(p.ld);
  uint32_t* hist = reinterpret_cast<uint32_t*>(dyn);
  uint32_t* cand = hist + 2 * S * 256;
  uint32_t* keys = cand + S * kCand;
  const int64_t r0 = int64_t(q) * p.Rc < R ? int64_t(q) * p.Rc : R;
  const int Rl = static_cast<int>((r0 + p.Rc < R ? r0 + p.Rc : R) - r0);  // this CTA's rows
  const int nparts = S < kKeyWarps ? kKeyWarps / S : 1;                      // warps per column in the statistics pass
  int64_t t_begin, t_end;
  split_range(p.T, gridDim.x / C, blockIdx.x / C, t_begin, t_end);
  uint32_t dor = 0, tor = 0;
  Emitter em;

  for (int64_t t = t_begin; t < t_end; ++t) {
    const int par = static_cast<int>(t & 1);
    const int64_t* dt = p.d + t * R * S;
    // ---- rank 0's values: the reference of every column's keys
    if (warp == 0) {
      int64_t x = lane < S ? __ldg(dt + lane) : 0;
      if (p.of_prefix) {
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int64_t up = __shfl_up_sync(kFull, x, o);
          if (lane >= o) x += up;
        }
      }
      if (lane < S) ks.ref[lane] = x;
    }
    __syncthreads();
    // ---- this CTA's rows -> keys
    bool bad = false;
    constexpr int kRows = (SC > 0 && SC <= 8) ? 2 : 1;  // rows in flight per thread
    for (int rl = tid; rl < Rl; rl += kRows * kKeyThreads) {
      const int64_t* row = dt + (r0 + rl) * S;
      bad |= store_row<SC>(p, row, S, ks, keys, rl, dor, tor);
      if (kRows == 2 && rl + kKeyThreads < Rl)
        bad |= store_row<SC>(p, row + kKeyThreads * S, S, ks, keys, rl + kKeyThreads, dor, tor);
    }
    const int cta_bad = __syncthreads_or(bad ? 1 : 0);
    // ---- column minimum, maximum and second largest key: `nparts` warps per column
    for (int item = warp; item < S * nparts; item += kKeyWarps) {
      const int s = item % S, part = item / S;
      const int a = Rl * part / nparts, b = Rl * (part + 1) / nparts;
      const uint32_t* col = keys + s * ld;
      uint32_t mn = 0xffffffffu, x1 = 0, x2 = 0;
      for (int rl = a + lane; rl < b; rl += 32) {
        const uint32_t k = col[rl];
        mn = k < mn ? k : mn;
        top2_merge<uint32_t>(x1, x2, k, 0u);
      }
      mn = __reduce_min_sync(kFull, mn);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const uint32_t o1 = __shfl_xor_sync(kFull, x1, o);
        const uint32_t o2 = __shfl_xor_sync(kFull, x2, o);
        top2_merge<uint32_t>(x1, x2, o1, o2);
      }
      if (lane == 0) {
        ks.pmn[item] = mn;
        ks.pmx[item] = x1;
        ks.psc[item] = x2;
      }
    }
    __syncthreads();
    if (tid < S) {
      uint32_t mn = 0xffffffffu, x1 = 0, x2 = 0;
      for (int item = tid; item < S * nparts; item += S) {
        mn = ks.pmn[item] < mn ? ks.pmn[item] : mn;
        top2_merge<uint32_t>(x1, x2, ks.pmx[item], ks.psc[item]);
      }
      ks.cmn[par][tid] = mn;
      ks.cmx[par][tid] = x1;
      ks.csc[par][tid] = x2;
    }
    if (tid == 32) ks.cbad[par] = static_cast<uint32_t>(cta_bad);
    cluster.sync();
    // ---- merge over the cluster (every CTA computes the same state)
    if (tid < S) {
      const int s = tid;
      uint32_t mn = 0xffffffffu, x1 = 0, x2 = 0;
      for (unsigned c = 0; c < C; ++c) {
        const KeyState* peer = cluster.map_shared_rank(&ks, c);
        const uint32_t pm = peer->cmn[par][s];
        mn = pm < mn ? pm : mn;
        top2_merge<uint32_t>(x1, x2, peer->cmx[par][s], peer->csc[par][s]);
      }
      const uint32_t range = x1 - mn;
      ks.lo[s] = mn;
      ks.nb[s] = range ? 32 - __clz(static_cast<int>(range)) : 0;
      ks.pref[s] = 0;
      ks.rem[s] = static_cast<uint32_t>((R - 1) / 2);
      ks.ncand[s] = 0;
      ks.compact[s] = 0;
      out.F[s] = key_value(ks.ref[s], x1);
      out.sec[s] = key_value(ks.ref[s], R >= 2 ? x2 : x1);
    } else if (tid == 32) {
      uint32_t b = 0;
      for (unsigned c = 0; c < C; ++c) b |= cluster.map_shared_rank(&ks, c)->cbad[par];
      ks.bad = b != 0;
    }
    __syncthreads();
    if (ks.bad) {
      // a value 2^31 or more away from rank 0's: the 64-bit path, by the cluster's first CTA
      if (q == 0) {
        select_step_lean(p, t, hist, g, out);
        if (warp == 0) em.step(p, t, out, lane);
      }
      continue;
    }
    int max_nb = 0;
    for (int s = 0; s < S; ++s) max_nb = ks.nb[s] > max_nb ? ks.nb[s] : max_nb;
    const int npass = (max_nb + 7) / 8;
    // ---- radix passes over the key offsets from the column minimum
    for (int j = 0; j < npass; ++j) {
      uint32_t* buf = hist + (j & 1) * S * 256;
      for (int i = tid; i < S * 64; i += kKeyThreads) reinterpret_cast<uint4*>(buf)[i] = make_uint4(0, 0, 0, 0);
      if (j == 1 && tid < S && ks.nb[tid] > 8) {
        // this CTA's count in the bin the first pass chose: its candidates for the later passes
        const int sh0 = ks.nb[tid] - 8;
        ks.compact[tid] = hist[tid * 256 + ((ks.pref[tid] >> sh0) & 255u)] <= kCand;
      }
      __syncthreads();
      for (int s = 0; s < S; ++s) {
        const int hi = ks.nb[s] - 8 * j;  // offset bits at and above `hi` are chosen
        if (hi <= 0) continue;
        const int sh = hi > 8 ? hi - 8 : 0;
        const uint32_t mask = (1u << (hi - sh)) - 1u, lo = ks.lo[s], pref = ks.pref[s];
        uint32_t* h = buf + s * 256;
        const uint32_t* col = keys + s * ld;
        if (j == 0) {
          // every key counts: four at a time
          const int nq = Rl >> 2;
          for (int i = tid; i < nq; i += kKeyThreads) {
            const uint4 k4 = reinterpret_cast<const uint4*>(col)[i];
            atomicAdd(&h[((k4.x - lo) >> sh) & mask], 1u);
            atomicAdd(&h[((k4.y - lo) >> sh) & mask], 1u);
            atomicAdd(&h[((k4.z - lo) >> sh) & mask], 1u);
            atomicAdd(&h[((k4.w - lo) >> sh) & mask], 1u);
          }
          for (int rl = 4 * nq + tid; rl < Rl; rl += kKeyThreads) atomicAdd(&h[((col[rl] - lo) >> sh) & mask], 1u);
        } else if (j == 1 && ks.compact[s]) {
          // count the matching keys and keep them as the column's candidates
          uint32_t* cs = cand + s * kCand;
          for (int base = warp * 32; base < Rl; base += kKeyThreads) {
            const int rl = base + lane;
            const uint32_t k = rl < Rl ? col[rl] : 0u;
            const uint32_t o = k - lo;
            const bool m = rl < Rl && (hi >= 32 || ((o ^ pref) >> hi) == 0);
            const uint32_t bal = __ballot_sync(kFull, m);
            if (bal) {
              uint32_t at = 0;
              if (lane == 0) at = atomicAdd(&ks.ncand[s], static_cast<uint32_t>(__popc(bal)));
              at = __shfl_sync(kFull, at, 0);
              if (m) {
                atomicAdd(&h[(o >> sh) & mask], 1u);
                cs[at + __popc(bal & ((1u << lane) - 1u))] = k;
              }
            }
          }
        } else if (j >= 2 && ks.compact[s]) {
          const uint32_t* cs = cand + s * kCand;
          const int n = static_cast<int>(ks.ncand[s]);
          for (int i = tid; i < n; i += kKeyThreads) {
            const uint32_t o = cs[i] - lo;
            if (hi >= 32 || ((o ^ pref) >> hi) == 0) atomicAdd(&h[(o >> sh) & mask], 1u);
          }
        } else {
          for (int rl = tid; rl < Rl; rl += kKeyThreads) {
            const uint32_t o = col[rl] - lo;
            if (hi >= 32 || ((o ^ pref) >> hi) == 0) atomicAdd(&h[(o >> sh) & mask], 1u);
          }
        }
      }
      cluster.sync();
      for (int s = warp; s < S; s += kKeyWarps) {
        const int hi = ks.nb[s] - 8 * j;
        if (hi <= 0) continue;
        uint32_t h[8] = {0, 0, 0, 0, 0, 0, 0, 0};
        // the cluster's histograms of the column, two CTAs' loads in flight at a time
        for (unsigned c0 = 0; c0 < C; c0 += 2) {
          uint4 a[2], b[2];
#pragma unroll
          for (int i = 0; i < 2; ++i) {
            if (c0 + i < C) {
              const uint4* pb = reinterpret_cast<const uint4*>(cluster.map_shared_rank(buf + s * 256, c0 + i));
              a[i] = pb[2 * lane];
              b[i] = pb[2 * lane + 1];
            }
          }
#pragma unroll
          for (int i = 0; i < 2; ++i) {
            if (c0 + i < C) {
              h[0] += a[i].x;
              h[1] += a[i].y;
              h[2] += a[i].z;
              h[3] += a[i].w;
              h[4] += b[i].x;
              h[5] += b[i].y;
              h[6] += b[i].z;
              h[7] += b[i].w;
            }
          }
        }
        uint32_t digit, below;
        bins_find(h, ks.rem[s], lane, digit, below);
        if (lane == 0) {
          ks.pref[s] |= digit << (hi > 8 ? hi - 8 : 0);
          ks.rem[s] -= below;
        }
      }
      __syncthreads();
    }
    if (tid < S) out.med[tid] = key_value(ks.ref[tid], ks.lo[tid] + ks.pref[tid]);
    __syncthreads();
    if (q == 0 && warp == 0) em.step(p, t, out, lane);
  }
  if (q == 0 && warp == 0) em.flush(p, lane);
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), p.of_prefix ? __reduce_or_sync(kFull, tor) : 0u);
  if (lane == 0) report(p.status, bits);
  cluster.sync();  // the cluster's other CTAs may still read this CTA's shared memory
}

template <int SC>
cudaError_t launch_keys(const RankParams& p, int C, size_t smem, cudaStream_t stream) {
  auto kern = rank_keys_kernel<SC>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(kKeyThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(C));
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg) != cudaSuccess || clusters < 1) {
    cudaGetLastError();
    clusters = std::max(1, sm_count() / C);
  }
  const int64_t n = std::min<int64_t>(clusters, p.T);
  cfg.gridDim = dim3(static_cast<unsigned>(n * C));
  count_launch();
  return cudaLaunchKernelEx(&cfg, kern, p);
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
  // smallest cluster whose shared memory holds the step's keys: first with
  // room for two CTAs per SM (one loads while the other selects), then one
  auto smem_for = [&](int C) {
    const int64_t rc = (R + C - 1) / C;
    return size_t(2 * S * 256 * 4) + size_t(S) * kCand * 4 + size_t(S) * size_t((rc + 3) & ~int64_t(3)) * 4;
  };
  int C = 0;
  for (size_t cap : {kRkSmemTwoPerSm, kRkSmemOnePerSm}) {
    for (int c = 1; c <= 8 && C == 0; c *= 2)
      if (smem_for(c) <= cap) C = c;
    if (C) break;
  }
  if (C) {
    p.Rc = (R + C - 1) / C;
    p.ld = (p.Rc + 3) & ~int64_t(3);
    const size_t smem = smem_for(C);
    switch (S) {
      case 4: return launch_keys<4>(p, C, smem, stream);
      case 6: return launch_keys<6>(p, C, smem, stream);
      case 8: return launch_keys<8>(p, C, smem, stream);
      case 10: return launch_keys<10>(p, C, smem, stream);
      case 16: return launch_keys<16>(p, C, smem, stream);
      default: return launch_keys<0>(p, C, smem, stream);
    }
  }
  // each CTA re-reads its current step once per byte of the range: keep the
  // steps in flight within about half of L2
  const int64_t sms = sm_count();
  const int64_t fit = std::max<int64_t>(sms, (int64_t(64) << 20) / (R * S * 8));
  const int grid = static_cast<int>(std::min<int64_t>(std::min<int64_t>(sms * 4, fit), T));
  count_launch();
  switch (S) {
    case 8: rank_global_kernel<8><<<grid, kRkThreads, 0, stream>>>(p); break;
    case 16: rank_global_kernel<16><<<grid, kRkThreads, 0, stream>>>(p); break;
    default: rank_global_kernel<0><<<grid, kRkThreads, 0, stream>>>(p); break;
  }
  return cudaGetLastError();
}

}  // namespace sf

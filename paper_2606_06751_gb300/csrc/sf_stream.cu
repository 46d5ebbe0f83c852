// sf_stream.cu - the streaming passes over the telemetry tensor d[T][R][S]:
//
//   * frontier pass (Sec. 3 Eq. 1-2): rank-local prefixes in registers, the
//     max-prefix frontier with its lowest attaining rank per boundary, the
//     increments a[t,s], and the fused window aggregation (X, D, E, C, leading
//     stage);
//   * evidence pass (Sec. 4 Eq. 4): the same frontier plus, for every stage s,
//     the makespan after replacing s by the clipped per-rank window median,
//     per-step leader confidence and the telemetry-quality sums (App. A);
//   * routing-baseline pass (Sec. 3 Props 1-2, Sec. 6): per-stage maxima and
//     sums, the slowest rank and rank 0 per window.
//
// Fast path (S even, S <= 16, R*S a multiple of 16): a persistent grid, one
// CTA per SM, each CTA owning a contiguous range of steps.  One producer
// thread streams 128-byte rows of d into a ring of shared-memory tiles with 2-D
// bulk tensor copies (TMA) completing on mbarriers; eight consumer warps read
// whole rank rows out of the tiles (128B-swizzled when S/2 is a power of two,
// which makes the strided 16-byte row reads bank-conflict free), keep the
// prefix and per-boundary maxima in registers, and reduce across ranks with
// warp redux plus one shared-memory exchange.  Small steps (<= 12 KB) are
// handled by one warp per tile of whole steps, each warp owning two ring
// stages; larger steps by one warp group per step, spread over one or more
// tiles, with two or four groups taking steps of one or two tiles in turn
// (each group owning its ring stages) and all eight warps on larger steps.
// The frontier over steps of up to 6 KB takes 2-8 steps per warp instruction
// (lanes_kernel: groups of lanes, one step each).  Fewer steps than SMs over
// many ranks split each step's ranks over a thread-block cluster
// (split_frontier_kernel).
//
// Generic path (any other S <= 32 or R): one CTA per step range with plain
// global loads.  All paths share the per-step epilogues.  A pass that follows
// the clear of its own outputs starts as that clear's programmatic dependent
// and writes only after griddep_wait().
#include <algorithm>
#include <array>
#include <numeric>
#include <type_traits>

#include <cooperative_groups.h>

#include "sf_device.cuh"
#include "sf_launch.h"

namespace sf {

namespace {

constexpr int kConsumerWarps = 8;
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kBlockThreads = kConsumerThreads + 32;  // + one producer warp
constexpr int kRowBytes = 128;                        // TMA row: 16 int64
// The 192 KB shared-memory ring is cut two ways.  Small steps (regime 0):
// 16 stages of 12 KB, two per consumer warp; warp w owns stages 2w and 2w+1
// and consumes every 8th tile through them in order, so no warp can run a
// phase ahead of a stage another warp still uses.  Large steps (regime 1):
// 6 stages of 32 KB that every consumer warp visits in order.
constexpr int kRingBytes = 192 * 1024;
constexpr int kR0Stages = 2 * kConsumerWarps;
constexpr int kR0StageBytes = kRingBytes / kR0Stages;  // 12 KB
constexpr int kR0MaxRows = kR0StageBytes / kRowBytes;   // 96 rows
constexpr int kR1Stages = 6;
constexpr int kR1StageBytes = kRingBytes / kR1Stages;  // 32 KB
constexpr int kR1MaxRows = kR1StageBytes / kRowBytes;   // 256 rows (the TMA box limit)
// The evidence pass streams the window medians m next to d (regime 1 only):
// 3 stages of 64 KB, each a 32 KB d tile and the matching 32 KB m tile.
constexpr int kR1GainStages = 3;
constexpr int kR1GainStageBytes = kRingBytes / kR1GainStages;  // 64 KB
constexpr int kR1GainMaxRows = kR1MaxRows;
constexpr int kMaxStages = kR0Stages;
constexpr int kRedPerWarp = 64;                       // per-warp partials of one step (<= 2S + 1)
constexpr int kRedSlots = 2 * kConsumerWarps * kRedPerWarp;  // double-buffered
constexpr size_t kSmemBytes = 1024 /*alignment slack*/ + size_t(kRingBytes) +
                              2 * kMaxStages * sizeof(uint64_t) + 16 + kRedSlots * sizeof(uint64_t);

struct Params {
  int64_t T, R, S;
  int64_t step_rows;  // 128-byte rows per step
  int regime;         // 0: several steps per tile, 1: tiles per step
  int box_rows, K, tiles_per_step;
  int64_t* a;
  int32_t* lead;
  int64_t* mk;
  int64_t* X;
  int64_t* D;
  int64_t* E;
  int32_t* C;
  uint8_t* step_lead;
  int64_t t0, W, w_first;
  const int64_t* m;
  const int64_t* wall;
  int other_stage;
  int64_t eta_num, eta_den;
  int64_t* Y;
  uint64_t* quality;
  uint32_t* status;
  int m_by_tma;  // evidence pass, regime 1: m tiles arrive through the ring
  int nst, stage_bytes;  // ring stages in use and their size
  int groups;            // regime 1: consumer warp groups, each taking every groups-th step
  // routing-baseline pass
  const int64_t* d;
  int64_t* bM;
  uint64_t* bSUM;
  int64_t* bSLOW;
  int64_t* bRANK0;
};

__device__ __forceinline__ uint32_t hi32(int64_t v) {
  return static_cast<uint32_t>(static_cast<uint64_t>(v) >> 32);
}

// --------------------------------------------------------------------------
// Window index of step t, (t0 + t) / W - w_first, recomputed (one 64-bit
// division) only when t passes the end of the last window seen: every thread
// visits its steps in increasing order, so that happens once per window
// rather than once per step.
struct WinTrack {
  int64_t lo = 0, hi = 0, w = 0;  // steps [lo, hi) belong to window w
  __device__ __forceinline__ int64_t at(int64_t t, int64_t t0, int64_t W, int64_t w_first) {
    if (t >= hi) {
      w = (t0 + t) / W - w_first;
      lo = (w + w_first) * W - t0;
      hi = lo + W;
    }
    return w;
  }
};

// Window accumulators held by the warp that finalizes steps: lane s keeps the
// stage-s numerators, every lane the denominator.
struct WinAcc {
  int64_t cur = -1;
  int64_t x = 0, y = 0, dsum = 0;
  int64_t erow = 0;  // E / C index of (window cur, this lane's stage, rank 0)
  WinTrack wt;
};

__device__ __forceinline__ void flush_window(const Params& p, int S, WinAcc& acc, int lane) {
  if (acc.cur >= 0) {
    if (lane < S) {
      if (acc.x) atomicAdd(reinterpret_cast<unsigned long long*>(&p.X[acc.cur * S + lane]),
                           static_cast<unsigned long long>(acc.x));
      if (p.Y && acc.y)
        atomicAdd(reinterpret_cast<unsigned long long*>(&p.Y[acc.cur * S + lane]),
                  static_cast<unsigned long long>(acc.y));
    }
    if (lane == 0 && acc.dsum)
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.D[acc.cur]),
                static_cast<unsigned long long>(acc.dsum));
  }
  acc.x = acc.y = acc.dsum = 0;
}

// Frontier epilogue for step t.  Lane s < S holds the packed key
// (F[t,s] << 16) | (65535 - lead[t,s]); the whole warp participates.
__device__ __forceinline__ void finalize_frontier(const Params& p, int S, int64_t t, uint64_t key,
                                                  int lane, WinAcc& acc) {
  const bool valid = lane < S;
  const int64_t F = valid ? static_cast<int64_t>(key >> 16) : 0;
  const int32_t ld = valid ? 65535 - static_cast<int32_t>(key & 0xffffu) : 0;
  int64_t Fprev = __shfl_up_sync(kFull, F, 1);
  if (lane == 0) Fprev = 0;  // F[t,-1] = 0
  const int64_t a = valid ? F - Fprev : 0;
  const int64_t mk = __shfl_sync(kFull, F, S - 1);
  if (valid) {
    if (p.a) p.a[t * S + lane] = a;
    if (p.lead) p.lead[t * S + lane] = ld;
  }
  if (lane == 0 && p.mk) p.mk[t] = mk;
  if (p.X) {
    const int64_t w = acc.wt.at(t, p.t0, p.W, p.w_first);
    if (w != acc.cur) {
      flush_window(p, S, acc, lane);
      acc.cur = w;
      acc.erow = (w * S + lane) * p.R;
    }
    acc.x += a;
    acc.dsum += mk;
    if (valid && ld >= 0 && ld < p.R) {  // always true for valid input; guards flagged input
      const int64_t idx = acc.erow + ld;
      if (p.E && a != 0)
        atomicAdd(reinterpret_cast<unsigned long long*>(&p.E[idx]), static_cast<unsigned long long>(a));
      if (p.C) atomicAdd(&p.C[idx], 1);
    }
    if (p.step_lead) {
      const uint64_t k2 = valid ? ((static_cast<uint64_t>(a) << 5) | static_cast<uint64_t>(31 - lane)) : 0;
      const uint64_t km = warp_max_u64(k2);
      if (lane == 0) p.step_lead[t] = static_cast<uint8_t>(31 - static_cast<int>(km & 31u));
    }
  }
}

// Evidence epilogue for step t.  Lane s < S holds the packed frontier key
// (F[t,s] << 16) | (65535 - lead[t,s]) and
// Fr[t,s] = max_r (P[t,r,S-1] - max(0, d[t,r,s] - m[w,r,s])).
__device__ __forceinline__ void finalize_gain(const Params& p, int S, int64_t t, uint64_t key,
                                              int64_t Fr, int lane, WinAcc& acc) {
  const bool valid = lane < S;
  const int64_t F = valid ? static_cast<int64_t>(key >> 16) : 0;
  const int32_t ld = valid ? 65535 - static_cast<int32_t>(key & 0xffffu) : 0;
  int64_t Fprev = __shfl_up_sync(kFull, F, 1);
  if (lane == 0) Fprev = 0;
  const int64_t a = valid ? F - Fprev : 0;
  const int64_t FS = __shfl_sync(kFull, F, S - 1);
  const int64_t y = valid ? FS - Fr : 0;
  // leading stage (largest increment, lowest stage) and the runner-up increment
  const uint64_t k2 = valid ? ((static_cast<uint64_t>(a) << 5) | static_cast<uint64_t>(31 - lane)) : 0;
  const uint64_t km = warp_max_u64(k2);
  const int best = 31 - static_cast<int>(km & 31u);
  const int64_t amax = static_cast<int64_t>(km >> 5);
  const int64_t second = static_cast<int64_t>(warp_max_u64(valid && lane != best ? static_cast<uint64_t>(a) : 0));
  const bool conf = FS > 0 && static_cast<__int128>(amax - second) * p.eta_den >=
                                  static_cast<__int128>(p.eta_num) * FS;
  if (lane == 0) p.step_lead[t] = static_cast<uint8_t>(best | (conf ? SF_STEP_CONFIDENT : 0u));
  const int64_t w = acc.wt.at(t, 0, p.W, 0);
  if (w != acc.cur) {
    flush_window(p, S, acc, lane);
    acc.cur = w;
    acc.erow = (w * S + lane) * p.R;
  }
  acc.x += a;
  acc.y += y;
  acc.dsum += FS;
  if (valid && ld >= 0 && ld < p.R) {  // lead-rank credit (always in range for valid input)
    const int64_t idx = acc.erow + ld;
    if (p.E && a != 0)
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.E[idx]), static_cast<unsigned long long>(a));
    if (p.C) atomicAdd(&p.C[idx], 1);
  }
}

// Routing-baseline window accumulators (lane s: stage s).
struct BaseAcc {
  int64_t cur = -1;
  int64_t m = 0, slow = 0, r0 = 0;
  unsigned __int128 sum = 0;
  WinTrack wt;
};

__device__ __forceinline__ void flush_base(const Params& p, int S, BaseAcc& acc, int lane) {
  if (acc.cur >= 0 && lane < S) {
    const int64_t i = acc.cur * S + lane;
    if (acc.m) atomicAdd(reinterpret_cast<unsigned long long*>(&p.bM[i]), static_cast<unsigned long long>(acc.m));
    if (acc.sum) atomic_add_u128(p.bSUM + 2 * i, acc.sum);
    if (acc.slow)
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.bSLOW[i]), static_cast<unsigned long long>(acc.slow));
    if (acc.r0) atomicAdd(reinterpret_cast<unsigned long long*>(&p.bRANK0[i]), static_cast<unsigned long long>(acc.r0));
  }
  acc.m = acc.slow = acc.r0 = 0;
  acc.sum = 0;
}

// Baseline epilogue for step t.  Lane s < S holds max_r d[t,r,s] and
// sum_r d[t,r,s]; every lane holds the packed key of the slowest rank
// (largest total, lowest rank on ties), whose row and rank 0's row are read
// back from d (the step was just streamed, so these hit L2).
__device__ __forceinline__ void finalize_base(const Params& p, int S, int64_t t, uint64_t mx, uint64_t sm,
                                              uint64_t slowkey, int lane, BaseAcc& acc) {
  const int64_t w = acc.wt.at(t, p.t0, p.W, p.w_first);
  if (w != acc.cur) {
    flush_base(p, S, acc, lane);
    acc.cur = w;
  }
  const int64_t rs = 65535 - static_cast<int64_t>(slowkey & 0xffffu);
  if (lane < S && rs >= 0 && rs < p.R) {  // always in range for valid input
    acc.m += static_cast<int64_t>(mx);
    acc.sum += sm;
    acc.slow += __ldg(p.d + (t * p.R + rs) * S + lane);
    acc.r0 += __ldg(p.d + t * p.R * S + lane);
  }
}

__device__ __forceinline__ uint64_t warp_sum_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

// Telemetry-quality sums of one thread (App. A closure / overlap), flushed per window.
struct QualAcc {
  int64_t cur = -1;
  unsigned __int128 res = 0, ovl = 0, wsum = 0;
};

__device__ __forceinline__ unsigned __int128 warp_sum_u128(unsigned __int128 v) {
  uint64_t lo = static_cast<uint64_t>(v), hi = static_cast<uint64_t>(v >> 64);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t olo = __shfl_xor_sync(kFull, lo, o);
    const uint64_t ohi = __shfl_xor_sync(kFull, hi, o);
    const uint64_t nlo = lo + olo;
    hi = hi + ohi + (nlo < lo ? 1u : 0u);
    lo = nlo;
  }
  return (static_cast<unsigned __int128>(hi) << 64) | lo;
}

// Warp-uniform: every lane calls with the same window index w.
__device__ __forceinline__ void qual_window(const Params& p, QualAcc& q, int64_t w, int lane) {
  if (w == q.cur) return;
  if (q.cur >= 0) {
    const unsigned __int128 r = warp_sum_u128(q.res), o = warp_sum_u128(q.ovl), s = warp_sum_u128(q.wsum);
    if (lane == 0) {
      uint64_t* dst = p.quality + q.cur * 6;
      if (r) atomic_add_u128(dst + 0, r);
      if (o) atomic_add_u128(dst + 2, o);
      if (s) atomic_add_u128(dst + 4, s);
    }
  }
  q.res = q.ovl = q.wsum = 0;
  q.cur = w;
}

__device__ __forceinline__ void qual_row(const Params& p, QualAcc& q, int64_t t, int64_t r,
                                         int64_t total, int64_t other, uint32_t& dor) {
  if (p.wall) {
    const int64_t wv = p.wall[t * p.R + r];
    dor |= hi32(wv);
    const int64_t e = wv - (total - other);  // e = w - sum_{s != other} d
    if (e > 0) q.res += static_cast<uint64_t>(e);
    else q.ovl += static_cast<uint64_t>(-e);
    q.wsum += static_cast<uint64_t>(wv);
  } else {
    q.res += static_cast<uint64_t>(other);
    q.wsum += static_cast<uint64_t>(total);
  }
}

// --------------------------------------------------------------------------
// Per-thread running maxima over the rank rows a thread visits (in increasing
// rank order, so a strict '>' keeps the lowest rank on ties).
template <int S>
struct FrontierRows {
  int64_t bp[S];
  int32_t br[S];
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int s = 0; s < S; ++s) {
      bp[s] = -1;
      br[s] = 0;
    }
  }
  __device__ __forceinline__ void row(const int64_t (&v)[S], int32_t r, uint32_t& dor, uint32_t& tor) {
    int64_t P = 0;
#pragma unroll
    for (int s = 0; s < S; ++s) {
      dor |= hi32(v[s]);
      P += v[s];  // P[t,r,s]
      if (P > bp[s]) {
        bp[s] = P;
        br[s] = r;
      }
    }
    tor |= hi32(P);
  }
  __device__ __forceinline__ uint64_t key(int s) const {
    return bp[s] < 0 ? 0ull
                     : (static_cast<uint64_t>(bp[s]) << 16) | static_cast<uint64_t>(65535 - br[s]);
  }
};

__host__ __device__ constexpr int ceil_log2(int x) { return x <= 1 ? 0 : 1 + ceil_log2((x + 1) / 2); }

// Evidence-pass maxima, with the frontier's lowest attaining rank.  A row
// whose durations and medians are all below 2^kNarrowBits
// (S * 2^kNarrowBits <= 2^31) is reduced in 32-bit arithmetic: its prefixes
// stay below 2^31 and P_S - d + m below 2^32, so every value is exact.  Other
// rows (long stages, invalid input) take the 64-bit path; the two partial
// maxima are merged at the end of the step.  Rows arrive in increasing rank
// order, so a strict '>' keeps the lowest rank on ties.
template <int S>
struct GainRows {
  static constexpr int kNarrowBits = 31 - ceil_log2(S);
  // With S > 10 the doubled state would spill; those shapes use the 64-bit path only.
  static constexpr bool kNarrow = S <= 10;
  uint32_t nf[S];        // narrow rows: 1 + max_r P[t,r,s] (0: none seen)
  int32_t nr[S];         //   and the lowest rank attaining it
  uint32_t ng[S];        //   max_r (P_S - max(0, d - m))
  int64_t bf[S];         // wide rows: max_r P (-1: none seen)
  int32_t br[S];
  int64_t bg[S];
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int s = 0; s < S; ++s) {
      nf[s] = ng[s] = 0;
      nr[s] = br[s] = 0;
      bf[s] = -1;
      bg[s] = 0;
    }
  }
  __device__ __forceinline__ int64_t row(const int64_t (&v)[S], const int64_t (&mr)[S], int32_t r, uint32_t& dor,
                                         uint32_t& tor) {
    uint32_t big = kNarrow ? 0u : 1u;
    if (kNarrow) {
#pragma unroll
      for (int s = 0; s < S; ++s)
        big |= hi32(v[s]) | hi32(mr[s]) |
               ((static_cast<uint32_t>(v[s]) | static_cast<uint32_t>(mr[s])) >> kNarrowBits);
    }
    if (big == 0) {
      uint32_t P1 = 1;  // prefix + 1
#pragma unroll
      for (int s = 0; s < S; ++s) {
        P1 += static_cast<uint32_t>(v[s]);
        if (P1 > nf[s]) {
          nf[s] = P1;
          nr[s] = r;
        }
      }
      const uint32_t P = P1 - 1;
#pragma unroll
      for (int s = 0; s < S; ++s) {
        // P_S - max(0, d - m) = min(P_S, P_S - d + m)
        const uint32_t alt = min(P, P - static_cast<uint32_t>(v[s]) + static_cast<uint32_t>(mr[s]));
        ng[s] = max(ng[s], alt);
      }
      return static_cast<int64_t>(P);
    }
    int64_t P = 0;
#pragma unroll
    for (int s = 0; s < S; ++s) {
      dor |= hi32(v[s]);
      P += v[s];
      if (P > bf[s]) {
        bf[s] = P;
        br[s] = r;
      }
    }
    tor |= hi32(P);
#pragma unroll
    for (int s = 0; s < S; ++s) {
      int64_t cut = v[s] - mr[s];
      cut = cut > 0 ? cut : 0;
      const int64_t alt = P - cut;
      bg[s] = alt > bg[s] ? alt : bg[s];
    }
    return P;
  }
  // packed (F << 16) | (65535 - lead); 0 when this thread saw no row
  __device__ __forceinline__ uint64_t key(int s) const {
    const uint64_t kn =
        nf[s] ? ((static_cast<uint64_t>(nf[s] - 1) << 16) | static_cast<uint64_t>(65535 - nr[s])) : 0ull;
    const uint64_t kw =
        bf[s] >= 0 ? ((static_cast<uint64_t>(bf[s]) << 16) | static_cast<uint64_t>(65535 - br[s])) : 0ull;
    return kn > kw ? kn : kw;
  }
  __device__ __forceinline__ uint64_t G(int s) const {
    const uint64_t w = static_cast<uint64_t>(bg[s]);
    return w > ng[s] ? w : static_cast<uint64_t>(ng[s]);
  }
};

// Routing-baseline maxima and sums over the rank rows a thread visits.
template <int S>
struct BaseRows {
  int64_t mx[S];
  uint64_t sm[S];
  uint64_t slow;  // (P_S << 16) | (65535 - r), max
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int s = 0; s < S; ++s) {
      mx[s] = 0;
      sm[s] = 0;
    }
    slow = 0;
  }
  __device__ __forceinline__ void row(const int64_t (&v)[S], int32_t r, uint32_t& dor, uint32_t& tor) {
    int64_t P = 0;
#pragma unroll
    for (int s = 0; s < S; ++s) {
      dor |= hi32(v[s]);
      P += v[s];
      mx[s] = v[s] > mx[s] ? v[s] : mx[s];
      sm[s] += static_cast<uint64_t>(v[s]);
    }
    tor |= hi32(P);
    const uint64_t k = (static_cast<uint64_t>(P) << 16) | static_cast<uint64_t>(65535 - r);
    slow = k > slow ? k : slow;
  }
};

template <int S>
__device__ __forceinline__ int64_t pick(const int64_t (&v)[S], int idx) {
  int64_t o = 0;
#pragma unroll
  for (int s = 0; s < S; ++s) o = (s == idx) ? v[s] : o;
  return o;
}

// Read rank row q (S int64) of a tile; the 16-byte chunk c of the tile lives
// at physical chunk c ^ ((c >> 3) & 7) when the tile was written with the
// 128-byte swizzle.
template <int S, bool kSwz>
__device__ __forceinline__ void load_row(const unsigned char* tile, int q, int64_t (&v)[S]) {
  constexpr int M = S / 2;
  const int c0 = q * M;
#pragma unroll
  for (int j = 0; j < M; ++j) {
    const int c = c0 + j;
    const int pc = kSwz ? (c ^ ((c >> 3) & 7)) : c;
    const longlong2 x = *reinterpret_cast<const longlong2*>(tile + pc * 16);
    v[2 * j] = x.x;
    v[2 * j + 1] = x.y;
  }
}

template <int S>
__device__ __forceinline__ void load_global_row(const int64_t* src, int64_t (&v)[S]) {
#pragma unroll
  for (int j = 0; j < S / 2; ++j) {
    const longlong2 x = __ldg(reinterpret_cast<const longlong2*>(src) + j);
    v[2 * j] = x.x;
    v[2 * j + 1] = x.y;
  }
}


// Ring stage and phase parity of the j-th tile a CTA streams.
// Regime 0: tile j belongs to warp j % 8, which alternates its two stages.
__device__ __forceinline__ void stage_of_r0(uint32_t j, uint32_t& st, uint32_t& ph) {
  const uint32_t i = j / kConsumerWarps;
  st = 2u * (j % kConsumerWarps) + (i & 1u);
  ph = (i >> 1) & 1u;
}

// Regime 1: the steps go to the warp groups in turn; group g owns stages g,
// g + G, ..., g + G (nst / G - 1) and fills them in that order.  The walk of
// one group's stages, kept incrementally (no division per tile).
struct GroupRing {
  uint32_t slot = 0, ph = 0;  // next stage slot within the group and its phase parity
  __device__ __forceinline__ uint32_t stage(uint32_t g, uint32_t G) const { return g + G * slot; }
  __device__ __forceinline__ void advance(uint32_t spg) {
    if (++slot == spg) {
      slot = 0;
      ph ^= 1u;
    }
  }
};


__device__ void produce(const CUtensorMap* map, const CUtensorMap* map_m, const Params& p, int64_t t_begin,
                        int64_t t_end, unsigned char* ring, uint64_t* full, uint64_t* empty,
                        volatile int* abort) {
  prefetch_tensormap(map);
  if (p.m_by_tma) prefetch_tensormap(map_m);
  const uint32_t bytes = static_cast<uint32_t>(p.box_rows) * kRowBytes;
  uint32_t j = 0;  // tiles issued
  uint32_t used = 0, last_ph = 0;  // per stage: issued into at all, parity of the last issue
  bool ok = true;
  auto issue = [&](int64_t row, int64_t mrow, uint32_t st, uint32_t ph) {
    if (!mbar_wait_bounded(&empty[st], ph ^ 1u, abort)) {
      ok = false;
      return;
    }
    used |= 1u << st;
    last_ph = (last_ph & ~(1u << st)) | (ph << st);
    unsigned char* dst = ring + size_t(st) * p.stage_bytes;
    mbar_arrive_expect_tx(&full[st], p.m_by_tma ? 2u * bytes : bytes);
    tma_load_2d(dst, map, 0, static_cast<int32_t>(row), &full[st]);
    if (p.m_by_tma) tma_load_2d(dst + p.stage_bytes / 2, map_m, 0, static_cast<int32_t>(mrow), &full[st]);
    ++j;
  };
  WinTrack mw;  // window of the medians streamed beside d (evidence pass)
  if (p.regime == 0) {
    for (int64_t t = t_begin; t < t_end && ok; t += p.K) {
      uint32_t st, ph;
      stage_of_r0(j, st, ph);
      issue(t * p.step_rows, 0, st, ph);
    }
  } else if (p.groups == 1) {
    GroupRing rg;
    const uint32_t nst = static_cast<uint32_t>(p.nst);
    for (int64_t t = t_begin; t < t_end && ok; ++t)
      for (int k = 0; k < p.tiles_per_step && ok; ++k) {
        const int64_t r0 = min(int64_t(k) * p.box_rows, p.step_rows - p.box_rows);
        issue(t * p.step_rows + r0, mw.at(t, 0, p.W, 0) * p.step_rows + r0, rg.slot, rg.ph);
        rg.advance(nst);
      }
  } else {
    const uint32_t G = static_cast<uint32_t>(p.groups), spg = static_cast<uint32_t>(p.nst) / G;
    uint32_t walk = 0;  // per group g (<= 4): bits 4g..4g+2 the next stage slot, bit 4g+3 its phase
    uint32_t g = 0;     // the group of step t
    for (int64_t t = t_begin; t < t_end && ok; ++t) {
      const uint32_t sh = 4u * g;
      uint32_t slot = (walk >> sh) & 7u, ph = (walk >> (sh + 3)) & 1u;
      for (int k = 0; k < p.tiles_per_step && ok; ++k) {
        const int64_t r0 = min(int64_t(k) * p.box_rows, p.step_rows - p.box_rows);
        issue(t * p.step_rows + r0, mw.at(t, 0, p.W, 0) * p.step_rows + r0, g + G * slot, ph);
        if (++slot == spg) {
          slot = 0;
          ph ^= 1u;
        }
      }
      walk = (walk & ~(15u << sh)) | (slot << sh) | (ph << (sh + 3));
      g = g + 1 == G ? 0 : g + 1;
    }
  }
  // copies still in flight: at most one per stage, the last issued into it
  for (uint32_t st = 0; st < kMaxStages; ++st)
    if ((used >> st) & 1u) mbar_wait_timeout(&full[st], (last_ph >> st) & 1u);
}

// --------------------------------------------------------------------------
// MODE 0: frontier (+ window aggregation); 1: evidence pass; 2: routing baselines.
template <int S, int MODE>
__global__ void __launch_bounds__(kBlockThreads, 1)
    stream_kernel(const __grid_constant__ CUtensorMap map, const __grid_constant__ CUtensorMap map_m,
                  const Params p) {
  constexpr bool GAIN = MODE == 1;
  constexpr bool BASE = MODE == 2;
  constexpr bool kSwz = (S == 4 || S == 8 || S == 16);
  constexpr int U = S <= 8 ? 4 : 2;  // rank rows in flight per thread
  extern __shared__ unsigned char smem_raw[];
  unsigned char* ring = align_1024(smem_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + kRingBytes);
  uint64_t* empty = full + kMaxStages;
  volatile int* abort = reinterpret_cast<volatile int*>(empty + kMaxStages);
  uint64_t* red = reinterpret_cast<uint64_t*>(empty + kMaxStages) + 2;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t G = gridDim.x, b = blockIdx.x;
  const int64_t t_begin = p.T * b / G, t_end = p.T * (b + 1) / G;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kMaxStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], p.regime == 0 ? 1u : uint32_t(kConsumerWarps / p.groups));
    }
    *abort = 0;
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kConsumerWarps) {
    if (lane == 0) produce(&map, &map_m, p, t_begin, t_end, ring, full, empty, abort);
    return;
  }
  griddep_wait();  // outputs cleared by the launch before this one (when it is its dependent)

  uint32_t dor = 0, tor = 0;  // OR of duration / rank-total high words
  WinAcc acc;
  QualAcc qa;
  WinTrack qt;  // window of the step a warp is on (evidence pass)
  BaseAcc bacc;
  const int R = static_cast<int>(p.R);

  if (p.regime == 0) {
    // ---- each warp owns every 8th tile (K whole steps) and two ring stages
    const int64_t n_local = t_end - t_begin;
    const int64_t n_tiles = (n_local + p.K - 1) / p.K;
    uint32_t i = 0;
    for (int64_t j = warp; j < n_tiles; j += kConsumerWarps, ++i) {
      const uint32_t st = 2u * warp + (i & 1u), ph = (i >> 1) & 1u;
      const bool have = mbar_wait_bounded(&full[st], ph, abort);
      const unsigned char* tile = ring + size_t(st) * kR0StageBytes;
      const int nsteps = static_cast<int>(min(int64_t(p.K), n_local - j * p.K));
      int kk0 = 0;
      if constexpr (MODE == 0 && S <= 8) {
        // frontier steps in pairs: two independent reduction chains per warp
        constexpr int UP = S <= 4 ? 2 : 1;  // rank rows of each step in flight per lane
        for (; kk0 + 1 < nsteps; kk0 += 2) {
          const int64_t t = t_begin + j * p.K + kk0;
          FrontierRows<S> ra, rb;
          ra.init();
          rb.init();
          if (have) {
            for (int r0 = lane; r0 < R; r0 += 32 * UP) {
              int64_t va[UP][S], vb[UP][S];
#pragma unroll
              for (int u = 0; u < UP; ++u)
                if (r0 + 32 * u < R) {
                  load_row<S, kSwz>(tile, kk0 * R + r0 + 32 * u, va[u]);
                  load_row<S, kSwz>(tile, (kk0 + 1) * R + r0 + 32 * u, vb[u]);
                }
#pragma unroll
              for (int u = 0; u < UP; ++u)
                if (r0 + 32 * u < R) {
                  ra.row(va[u], r0 + 32 * u, dor, tor);
                  rb.row(vb[u], r0 + 32 * u, dor, tor);
                }
            }
          }
          uint64_t ka = 0, kb = 0;
#pragma unroll
          for (int s = 0; s < S; ++s) {
            const uint64_t ma = warp_max_u64(ra.key(s));
            const uint64_t mb = warp_max_u64(rb.key(s));
            if (lane == s) {
              ka = ma;
              kb = mb;
            }
          }
          finalize_frontier(p, S, t, ka, lane, acc);
          finalize_frontier(p, S, t + 1, kb, lane, acc);
        }
      }
      for (int kk = kk0; kk < nsteps; ++kk) {
        const int64_t t = t_begin + j * p.K + kk;
        const int64_t w = GAIN ? qt.at(t, 0, p.W, 0) : 0;
        if (GAIN && p.quality) qual_window(p, qa, w, lane);
        const int q0 = kk * R;
        if constexpr (MODE == 0) {
          FrontierRows<S> rs;
          rs.init();
          if (have) {
            for (int r0 = lane; r0 < R; r0 += 32 * U) {
              int64_t v[U][S];
#pragma unroll
              for (int u = 0; u < U; ++u)
                if (r0 + 32 * u < R) load_row<S, kSwz>(tile, q0 + r0 + 32 * u, v[u]);
#pragma unroll
              for (int u = 0; u < U; ++u)
                if (r0 + 32 * u < R) rs.row(v[u], r0 + 32 * u, dor, tor);
            }
          }
          uint64_t mykey = 0;
#pragma unroll
          for (int s = 0; s < S; ++s) {
            const uint64_t km = warp_max_u64(rs.key(s));
            if (lane == s) mykey = km;
          }
          finalize_frontier(p, S, t, mykey, lane, acc);
        } else if constexpr (BASE) {
          BaseRows<S> rs;
          rs.init();
          if (have) {
            for (int r0 = lane; r0 < R; r0 += 32 * U) {
              int64_t v[U][S];
#pragma unroll
              for (int u = 0; u < U; ++u)
                if (r0 + 32 * u < R) load_row<S, kSwz>(tile, q0 + r0 + 32 * u, v[u]);
#pragma unroll
              for (int u = 0; u < U; ++u)
                if (r0 + 32 * u < R) rs.row(v[u], r0 + 32 * u, dor, tor);
            }
          }
          uint64_t myM = 0, mySum = 0;
#pragma unroll
          for (int s = 0; s < S; ++s) {
            const uint64_t mx = warp_max_u64(static_cast<uint64_t>(rs.mx[s]));
            const uint64_t sm = warp_sum_u64(rs.sm[s]);
            if (lane == s) {
              myM = mx;
              mySum = sm;
            }
          }
          finalize_base(p, S, t, myM, mySum, warp_max_u64(rs.slow), lane, bacc);
        } else {
          GainRows<S> rs;
          rs.init();
          if (have) {
            for (int r = lane; r < R; r += 32) {
              int64_t v[S], mr[S];
              load_row<S, kSwz>(tile, q0 + r, v);
              load_global_row<S>(p.m + (w * p.R + r) * S, mr);
              const int64_t total = rs.row(v, mr, r, dor, tor);
              if (p.quality)
                qual_row(p, qa, t, r, total, p.other_stage >= 0 ? pick<S>(v, p.other_stage) : 0, dor);
            }
          }
          uint64_t myK = 0;
          int64_t myR = 0;
#pragma unroll
          for (int s = 0; s < S; ++s) {
            const uint64_t f = warp_max_u64(rs.key(s));
            const uint64_t g = warp_max_u64(rs.G(s));
            if (lane == s) {
              myK = f;
              myR = static_cast<int64_t>(g);
            }
          }
          finalize_gain(p, S, t, myK, myR, lane, acc);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }
  } else {
    // ---- one step per warp group (of kConsumerWarps / groups warps), the
    // groups taking steps in turn, tiles_per_step tiles per step
    // (the group count is a compile-time constant in each copy of the loop)
    auto consume = [&](auto ng) {
      constexpr int NG = decltype(ng)::value;
      constexpr int gw = kConsumerWarps / NG;  // warps per group
      const int g = warp / gw, lw = warp % gw;
      constexpr int gthreads = gw * 32;
      const int ctid = threadIdx.x - g * gthreads;  // thread within the group
      const uint32_t spg = static_cast<uint32_t>(p.nst / NG);  // stages of this group
      GroupRing gring;
      int buf = 0;
      for (int64_t t = t_begin + g; t < t_end; t += NG) {
        const int64_t w = GAIN ? qt.at(t, 0, p.W, 0) : 0;
        if (GAIN && p.quality) qual_window(p, qa, w, lane);
        [[maybe_unused]] FrontierRows<S> fr;
        [[maybe_unused]] GainRows<S> gr;
        [[maybe_unused]] BaseRows<S> br;
        if constexpr (GAIN) gr.init();
        else if constexpr (BASE) br.init();
        else fr.init();
        for (int k = 0; k < p.tiles_per_step; ++k) {
          const uint32_t st = gring.stage(g, NG), ph = gring.ph;
          gring.advance(spg);
          const bool have = mbar_wait_bounded(&full[st], ph, abort);
          const unsigned char* tile = ring + size_t(st) * p.stage_bytes;
          const int64_t row0 = min(int64_t(k) * p.box_rows, p.step_rows - p.box_rows);
          const int rank_tile0 = static_cast<int>(row0 * 16 / S);
          const int rank_fresh = static_cast<int>(int64_t(k) * p.box_rows * 16 / S);
          const int rank_end = static_cast<int>((row0 + p.box_rows) * 16 / S);
          if (have) {
            if constexpr (!GAIN) {
              for (int r0 = rank_fresh + ctid; r0 < rank_end; r0 += gthreads * U) {
                int64_t v[U][S];
  #pragma unroll
                for (int u = 0; u < U; ++u)
                  if (r0 + gthreads * u < rank_end) load_row<S, kSwz>(tile, r0 + gthreads * u - rank_tile0, v[u]);
  #pragma unroll
                for (int u = 0; u < U; ++u)
                  if (r0 + gthreads * u < rank_end) {
                    if constexpr (BASE) br.row(v[u], r0 + gthreads * u, dor, tor);
                    else fr.row(v[u], r0 + gthreads * u, dor, tor);
                  }
              }
            } else {
              constexpr int UG = 1;  // rank rows in flight per thread
              for (int r0 = rank_fresh + ctid; r0 < rank_end; r0 += gthreads * UG) {
                int64_t v[UG][S], mr[UG][S];
  #pragma unroll
                for (int u = 0; u < UG; ++u)
                  if (r0 + gthreads * u < rank_end) {
                    const int q = r0 + gthreads * u - rank_tile0;
                    load_row<S, kSwz>(tile, q, v[u]);
                    load_row<S, kSwz>(tile + p.stage_bytes / 2, q, mr[u]);  // m tile of the same ranks
                  }
  #pragma unroll
                for (int u = 0; u < UG; ++u)
                  if (r0 + gthreads * u < rank_end) {
                    const int r = r0 + gthreads * u;
                    const int64_t total = gr.row(v[u], mr[u], r, dor, tor);
                    if (p.quality)
                      qual_row(p, qa, t, r, total, p.other_stage >= 0 ? pick<S>(v[u], p.other_stage) : 0, dor);
                  }
              }
            }
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&empty[st]);
        }
        // cross-rank reduction: warp redux, then one exchange through shared memory
        uint64_t* slot = red + (buf * kConsumerWarps + warp) * kRedPerWarp;
        uint64_t bslow = 0;
        if constexpr (BASE) bslow = warp_max_u64(br.slow);
  #pragma unroll
        for (int s = 0; s < S; ++s) {
          if constexpr (MODE == 0) {
            const uint64_t km = warp_max_u64(fr.key(s));
            if (lane == s) slot[s] = km;
          } else if constexpr (BASE) {
            const uint64_t mx = warp_max_u64(static_cast<uint64_t>(br.mx[s]));
            const uint64_t sm = warp_sum_u64(br.sm[s]);
            if (lane == s) {
              slot[s] = mx;
              slot[S + s] = sm;
            }
          } else {
            const uint64_t f = warp_max_u64(gr.key(s));
            const uint64_t g = warp_max_u64(gr.G(s));
            if (lane == s) {
              slot[s] = f;
              slot[S + s] = g;
            }
          }
        }
        if (BASE && lane == 0) slot[2 * S] = bslow;
        // the group's own barrier, its id an immediate operand
        switch (g) {
          case 0: named_barrier(1, gthreads); break;
          case 1: named_barrier(2, gthreads); break;
          case 2: named_barrier(3, gthreads); break;
          default: named_barrier(4, gthreads); break;
        }
        if (lw == 0) {
          uint64_t v0 = 0, v1 = 0, v2 = 0;
          if (lane < S) {
            for (int ww = warp; ww < warp + gw; ++ww) {
              const uint64_t* sl = red + (buf * kConsumerWarps + ww) * kRedPerWarp;
              v0 = sl[lane] > v0 ? sl[lane] : v0;
              if (GAIN) v1 = sl[S + lane] > v1 ? sl[S + lane] : v1;
              if (BASE) v1 += sl[S + lane];
            }
          }
          if (BASE) {
            for (int ww = warp; ww < warp + gw; ++ww) {
              const uint64_t k = red[(buf * kConsumerWarps + ww) * kRedPerWarp + 2 * S];
              v2 = k > v2 ? k : v2;
            }
          }
          if constexpr (MODE == 0) finalize_frontier(p, S, t, v0, lane, acc);
          else if constexpr (BASE) finalize_base(p, S, t, v0, v1, v2, lane, bacc);
          else finalize_gain(p, S, t, v0, static_cast<int64_t>(v1), lane, acc);
        }
        buf ^= 1;
      }
    };
    if (p.groups == 4) consume(std::integral_constant<int, 4>{});
    else if (p.groups == 2) consume(std::integral_constant<int, 2>{});
    else consume(std::integral_constant<int, 1>{});
  }

  const bool leader = p.regime == 0 || warp % (kConsumerWarps / p.groups) == 0;  // holds window accumulators
  if (BASE && leader) flush_base(p, S, bacc, lane);
  if (!BASE && p.X && leader) flush_window(p, S, acc, lane);
  if (GAIN && p.quality) qual_window(p, qa, -2, lane);
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), __reduce_or_sync(kFull, tor)) |
                        (*abort ? SF_ST_TIMEOUT : 0u);
  if (lane == 0) report(p.status, bits);
}

// --------------------------------------------------------------------------
// Frontier pass over small steps (R*S <= 768, S in {2, 4, 8, 16}): G steps
// share each warp instruction.  A warp splits into G groups of L = 32 / G
// lanes; group g takes step kk0 + g of the warp's tile and lane j of the group
// visits ranks j, j + L, ... in increasing order, so a strict '>' keeps the
// lowest rank within a lane.  The per-stage packed keys (F << 16 | 65535 - r)
// are then reduced over the group's L lanes by exchanges that halve the set of
// keys a lane holds at each step (G steps' reductions in the instructions of
// one), and the lanes j < S of each group run the step's epilogue for their
// own step, so the per-step epilogue cost is shared by G steps as well.  The
// tiles (K whole steps, K a multiple of G) arrive through the same warp-owned
// ring stages as the other small-step path, from the same producer.  With
// consecutive ranks in consecutive lanes, the 128-byte swizzle places the 16
// or 8 lanes of a group on distinct 16-byte bank groups, so a group's row
// reads are conflict free.
template <int S, int L>
__device__ __forceinline__ uint64_t group_max_keys(uint64_t (&k)[S], int j) {
  static_assert(L >= S && (S & (S - 1)) == 0 && (L & (L - 1)) == 0, "L >= S, both powers of two");
#pragma unroll
  for (int lvl = 0; (L >> (lvl + 1)) >= 1; ++lvl) {
    const int o = L >> (lvl + 1);
    const int n = S >> lvl;  // keys this lane still holds
    if (n > 1) {
      // the lane with bit o set keeps the upper half of its keys, its partner the lower
      const bool up = (j & o) != 0;
#pragma unroll
      for (int i = 0; i < n / 2; ++i) {
        const uint64_t send = up ? k[i] : k[i + n / 2];
        const uint64_t keep = up ? k[i + n / 2] : k[i];
        const uint64_t got = __shfl_xor_sync(kFull, send, o);
        k[i] = keep > got ? keep : got;
      }
    } else {
      const uint64_t got = __shfl_xor_sync(kFull, k[0], o);
      k[0] = k[0] > got ? k[0] : got;
    }
  }
  // lane j now holds the group maximum of stage j >> (log2 L - log2 S)
  return k[0];
}

// Frontier epilogue of one group's step t (the group's lanes j < S hold the
// packed keys of stages j); the whole warp calls it, live = false for groups
// past the tile's last step.
template <int S, int L>
__device__ __forceinline__ void finalize_group(const Params& p, int64_t t, uint64_t key, int j, bool live,
                                               WinAcc& acc) {
  const bool valid = live && j < S;
  const int64_t F = valid ? static_cast<int64_t>(key >> 16) : 0;
  const int32_t ld = valid ? 65535 - static_cast<int32_t>(key & 0xffffu) : 0;
  int64_t Fprev = __shfl_up_sync(kFull, F, 1, L);
  if (j == 0) Fprev = 0;  // F[t,-1] = 0
  const int64_t a = valid ? F - Fprev : 0;
  const int64_t mk = __shfl_sync(kFull, F, S - 1, L);
  uint64_t km = 0;
  if (p.X && p.step_lead) {
    // leading stage: largest increment, lowest stage on ties
    km = valid ? ((static_cast<uint64_t>(a) << 5) | static_cast<uint64_t>(31 - j)) : 0;
#pragma unroll
    for (int o = 1; o < S; o <<= 1) {
      const uint64_t got = __shfl_xor_sync(kFull, km, o);
      km = km > got ? km : got;
    }
  }
  if (!live) return;
  if (valid) {
    if (p.a) p.a[t * S + j] = a;
    if (p.lead) p.lead[t * S + j] = ld;
  }
  if (j == 0 && p.mk) p.mk[t] = mk;
  if (p.X) {
    const int64_t w = acc.wt.at(t, p.t0, p.W, p.w_first);
    if (w != acc.cur) {
      flush_window(p, S, acc, j);
      acc.cur = w;
      acc.erow = (w * S + j) * p.R;
    }
    acc.x += a;
    acc.dsum += mk;
    if (valid && ld >= 0 && ld < p.R) {  // always true for valid input; guards flagged input
      const int64_t idx = acc.erow + ld;
      if (p.E && a != 0)
        atomicAdd(reinterpret_cast<unsigned long long*>(&p.E[idx]), static_cast<unsigned long long>(a));
      if (p.C) atomicAdd(&p.C[idx], 1);
    }
    if (p.step_lead && j == 0) p.step_lead[t] = static_cast<uint8_t>(31 - static_cast<int>(km & 31u));
  }
}

template <int S, int G>
__global__ void __launch_bounds__(kBlockThreads, 1)
    lanes_kernel(const __grid_constant__ CUtensorMap map, const Params p) {
  constexpr int L = 32 / G;
  constexpr int U = S <= 8 ? 4 : 2;  // rank rows in flight per lane
  constexpr int kShift = ceil_log2(L) - ceil_log2(S);
  extern __shared__ unsigned char smem_raw[];
  unsigned char* ring = align_1024(smem_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + kRingBytes);
  uint64_t* empty = full + kMaxStages;
  volatile int* abort = reinterpret_cast<volatile int*>(empty + kMaxStages);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t NB = gridDim.x, b = blockIdx.x;
  const int64_t t_begin = p.T * b / NB, t_end = p.T * (b + 1) / NB;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kMaxStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    *abort = 0;
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kConsumerWarps) {
    if (lane == 0) produce(&map, &map, p, t_begin, t_end, ring, full, empty, abort);
    return;
  }
  griddep_wait();  // outputs cleared by the launch before this one (when it is its dependent)

  const int g = lane / L, j = lane % L;
  uint32_t dor = 0, tor = 0;
  WinAcc acc;
  const int R = static_cast<int>(p.R);
  const int64_t n_local = t_end - t_begin;
  const int64_t n_tiles = (n_local + p.K - 1) / p.K;
  // one round: group g takes step kk of `tile` (step t of the pass)
  auto round = [&](const unsigned char* tile, int kk, int64_t t, bool live, bool have) {
    FrontierRows<S> rs;
    rs.init();
    if (have && live) {
      const int q0 = kk * R;
      for (int r0 = j; r0 < R; r0 += L * U) {
        int64_t v[U][S];
#pragma unroll
        for (int u = 0; u < U; ++u)
          if (r0 + L * u < R) load_row<S, true>(tile, q0 + r0 + L * u, v[u]);
#pragma unroll
        for (int u = 0; u < U; ++u)
          if (r0 + L * u < R) rs.row(v[u], r0 + L * u, dor, tor);
      }
    }
    uint64_t k[S];
#pragma unroll
    for (int s = 0; s < S; ++s) k[s] = rs.key(s);
    const uint64_t ks = group_max_keys<S, L>(k, j);
    // lane j < S of the group takes stage j's key from the lane holding it
    const uint64_t mykey = __shfl_sync(kFull, ks, (j & (S - 1)) << kShift, L);
    finalize_group<S, L>(p, t, mykey, j, live, acc);
  };
  // K steps per tile (a multiple of G): the warp's tiles one at a time, G steps per round
  uint32_t i = 0;
  for (int64_t jt = warp; jt < n_tiles; jt += kConsumerWarps, ++i) {
    const uint32_t st = 2u * warp + (i & 1u), ph = (i >> 1) & 1u;
    const bool have = mbar_wait_bounded(&full[st], ph, abort);
    const unsigned char* tile = ring + size_t(st) * p.stage_bytes;
    const int nsteps = static_cast<int>(min(int64_t(p.K), n_local - jt * p.K));
    for (int kk0 = 0; kk0 < nsteps; kk0 += G) {
      const int kk = kk0 + g;
      round(tile, kk, t_begin + jt * p.K + kk, kk < nsteps, have);
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[st]);
  }

  if (p.X) flush_window(p, S, acc, j);
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), __reduce_or_sync(kFull, tor)) |
                        (*abort ? SF_ST_TIMEOUT : 0u);
  if (lane == 0) report(p.status, bits);
}

// Steps per warp instruction of the small-step frontier pass: the largest
// G in {2, 4, 8} with L = 32 / G >= S and G whole steps in one ring stage;
// 0 when the shape takes the one-step-per-warp path.  (Steps of 6-12 KB,
// one per stage, stay there: a warp taking both of its stages in one round
// has no copy of its own in flight, and the in-order producer then holds
// every warp up; measured at less than half the one-step-per-warp rate.)
int lanes_groups(int64_t R, int64_t S) {
  if (S != 2 && S != 4 && S != 8 && S != 16) return 0;
  const int64_t step_rows = R * S / 16;
  int G = 0;
  for (int c = 2; c <= 8; c *= 2)
    if (32 / c >= S && c * step_rows <= kR0MaxRows) G = c;
  return G;
}

// --------------------------------------------------------------------------
// Few steps over many ranks (fewer steps than SMs: one window of a few
// hundred steps, the per-window use of Sec. 3): each step's ranks are split
// over a thread-block cluster of `csize` CTAs, so every SM streams.  CTA j of
// the cluster reads ranks [j R / csize, (j+1) R / csize) with 16-byte loads
// (four rows in flight per thread), reduces its packed per-stage keys
// (F << 16 | 65535 - r) to shared memory, and the cluster's first CTA takes
// the maximum over the cluster's keys through distributed shared memory
// (ranks are disjoint, so the largest key still carries the lowest attaining
// rank) and runs the step's epilogue.  No global scratch.
constexpr int kSplitThreads = 256;
constexpr int kSplitMaxCluster = 16;  // above 8: a non-portable cluster size, allowed per kernel

template <int S>
__global__ void __launch_bounds__(kSplitThreads) split_frontier_kernel(const int64_t* __restrict__ d, const Params p) {
  namespace cg = cooperative_groups;
  cg::cluster_group cl = cg::this_cluster();
  __shared__ uint64_t wkey[kSplitThreads / 32][S];
  __shared__ uint64_t ckey[S];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int csize = static_cast<int>(cl.num_blocks());
  const int j = static_cast<int>(cl.block_rank());
  const int64_t t = blockIdx.x / csize;
  const int64_t R = p.R;
  const int64_t r0 = R * j / csize, r1 = R * (j + 1) / csize;
  const int64_t* dt = d + t * R * S;
  FrontierRows<S> fr;
  fr.init();
  uint32_t dor = 0, tor = 0;
  constexpr int U = 4;
  for (int64_t r = r0 + threadIdx.x; r < r1; r += int64_t(kSplitThreads) * U) {
    int64_t v[U][S];
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (r + int64_t(kSplitThreads) * u < r1) load_global_row<S>(dt + (r + int64_t(kSplitThreads) * u) * S, v[u]);
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (r + int64_t(kSplitThreads) * u < r1) fr.row(v[u], static_cast<int32_t>(r + kSplitThreads * u), dor, tor);
  }
#pragma unroll
  for (int s = 0; s < S; ++s) {
    const uint64_t km = warp_max_u64(fr.key(s));
    if (lane == 0) wkey[warp][s] = km;
  }
  __syncthreads();
  if (threadIdx.x < S) {
    uint64_t k = 0;
    for (int w = 0; w < kSplitThreads / 32; ++w) k = wkey[w][threadIdx.x] > k ? wkey[w][threadIdx.x] : k;
    ckey[threadIdx.x] = k;
  }
  cl.sync();  // every CTA's keys are visible to the cluster
  if (j == 0 && warp == 0) {
    griddep_wait();  // outputs cleared by the launch before this one (when it is its dependent)
    uint64_t key = 0;
    if (lane < S)
      for (int q = 0; q < csize; ++q) {
        const uint64_t k = *cl.map_shared_rank(&ckey[lane], static_cast<unsigned>(q));
        key = k > key ? k : key;
      }
    WinAcc acc;
    finalize_frontier(p, S, t, key, lane, acc);
    if (p.X) flush_window(p, S, acc, lane);
  }
  cl.sync();  // the other CTAs' shared memory stays alive until the first CTA has read it
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), __reduce_or_sync(kFull, tor));
  if (lane == 0) report(p.status, bits);
}

template <int S>
cudaError_t launch_split(const int64_t* d, const Params& p, int csize, cudaStream_t stream, bool pdl) {
  static bool ready = false;  // attribute set once per process (same on every GB300)
  if (!ready) {
    const cudaError_t e = cudaFuncSetAttribute(split_frontier_kernel<S>,
                                               cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    ready = true;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(csize);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see launch_ex
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(p.T * csize));
  cfg.blockDim = dim3(kSplitThreads);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, split_frontier_kernel<S>, d, p);
}

// Cluster size for T steps over R ranks: the largest size (<= 16, at least
// 512 ranks per CTA) at which all T clusters are resident at once.  A
// cluster is placed within one GPC, so sizes that do not divide a GPC's CTA
// slots evenly fit fewer clusters than the SM count suggests, and a second
// wave of clusters costs more than the parallelism gained (100 steps x 8192
// ranks: 1, 3, 6 and 12 CTAs per step ran at 20.6, 21.9, 25.0 and 28.3 us).
// The resident counts come from the occupancy calculator, once per process.
template <int S>
int split_cluster_size(int64_t T, int64_t R) {
  static const std::array<int, kSplitMaxCluster + 1> fit = [] {
    std::array<int, kSplitMaxCluster + 1> f{};
    if (cudaFuncSetAttribute(split_frontier_kernel<S>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
        cudaSuccess) {
      cudaGetLastError();
      return f;
    }
    for (int c = 1; c <= kSplitMaxCluster; ++c) {
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = static_cast<unsigned>(c);
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.gridDim = dim3(static_cast<unsigned>(c));
      cfg.blockDim = dim3(kSplitThreads);
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, split_frontier_kernel<S>, &cfg) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
      }
      f[c] = n;
    }
    return f;
  }();
  int best = 1;
  for (int c = 2; c <= kSplitMaxCluster; ++c)
    if (R / c >= 512 && fit[c] >= T) best = c;
  return best;
}

int split_cluster(int S, int64_t T, int64_t R) {
  switch (S) {
    case 2: return split_cluster_size<2>(T, R);
    case 4: return split_cluster_size<4>(T, R);
    case 6: return split_cluster_size<6>(T, R);
    case 8: return split_cluster_size<8>(T, R);
    case 10: return split_cluster_size<10>(T, R);
    case 12: return split_cluster_size<12>(T, R);
    case 14: return split_cluster_size<14>(T, R);
    case 16: return split_cluster_size<16>(T, R);
    default: return 1;
  }
}

cudaError_t dispatch_split(int S, const int64_t* d, const Params& p, int csize, cudaStream_t stream, bool pdl) {
  switch (S) {
    case 2: return launch_split<2>(d, p, csize, stream, pdl);
    case 4: return launch_split<4>(d, p, csize, stream, pdl);
    case 6: return launch_split<6>(d, p, csize, stream, pdl);
    case 8: return launch_split<8>(d, p, csize, stream, pdl);
    case 10: return launch_split<10>(d, p, csize, stream, pdl);
    case 12: return launch_split<12>(d, p, csize, stream, pdl);
    case 14: return launch_split<14>(d, p, csize, stream, pdl);
    case 16: return launch_split<16>(d, p, csize, stream, pdl);
    default: return cudaErrorInvalidValue;
  }
}

// --------------------------------------------------------------------------
// Untiled bulk copy global -> shared (both 16-byte aligned, a multiple of 16
// bytes), completion counted in bytes on `bar`.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

// Orders this CTA's earlier shared-memory accesses (generic proxy) before
// later bulk copies into shared memory (async proxy).
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Generic path: any S <= 32, any R; one CTA of 256 threads per step range.
// The per-stage state is sized by the bound SMAX >= S (4, 8, 16 or 32) and
// every stage loop is unrolled to SMAX with an `s < S` guard, so the state
// stays in registers.
constexpr int kGenThreads = 256;

// RING: the CTA's steps are one contiguous byte range of d, streamed with
// bulk copies in kGenRingStages chunks of p.stage_bytes (a power of two) into
// a shared-memory ring; rows are read from the ring at their offset in that
// range (a row may straddle chunks), and only a row past the range's last
// 16-byte boundary is read from global memory.  Thread 0 refills the chunks
// the finished step no longer needs right after the step's closing barrier,
// so no stage is overwritten while a thread still reads it.  A step must fit
// in kGenRingStages - 1 chunks (checked by the host).
constexpr uint32_t kGenRingStages = 8;

template <int SMAX, int MODE, bool VEC, bool RING>
__global__ void __launch_bounds__(kGenThreads)
    stream_generic_kernel(const int64_t* __restrict__ d, const Params p) {
  constexpr bool GAIN = MODE == 1;
  constexpr bool BASE = MODE == 2;
  constexpr uint32_t NST = kGenRingStages;
  __shared__ uint64_t red[kGenThreads / 32][66];
  __shared__ uint64_t full[RING ? NST : 1];
  __shared__ int abort_word;
  extern __shared__ __align__(128) unsigned char ring[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = static_cast<int>(p.S);
  const int64_t R = p.R;
  const int64_t G = gridDim.x, b = blockIdx.x;
  const int64_t t_begin = p.T * b / G, t_end = p.T * (b + 1) / G;
  uint32_t dor = 0, tor = 0;
  WinAcc acc;
  QualAcc qa;
  WinTrack qt;  // window of the step a warp is on (evidence pass)
  BaseAcc bacc;
  // ring geometry (RING only): bytes [A0, B0) of d, chunk c in stage c % NST
  const int64_t RS8 = R * S * 8;
  const uint32_t CB = static_cast<uint32_t>(p.stage_bytes);
  const uint32_t cshift = RING ? static_cast<uint32_t>(__ffs(static_cast<int>(CB)) - 1) : 0u;
  const uint32_t RBmask = NST * CB - 1;
  const int64_t A0 = (t_begin * RS8) & ~int64_t(15), B0 = (t_end * RS8) & ~int64_t(15);
  const int64_t nchunks = RING && B0 > A0 ? (B0 - A0 + CB - 1) >> cshift : 0;
  const unsigned char* dbytes = reinterpret_cast<const unsigned char*>(d);
  volatile int* abort = &abort_word;
  int64_t issued = 0, released = 0;  // thread 0: chunks issued; chunks no step needs any more
  auto issue = [&](int64_t c) {
    const uint32_t st = static_cast<uint32_t>(c) & (NST - 1);
    const int64_t off = A0 + (c << cshift);
    const uint32_t bytes = static_cast<uint32_t>(min(int64_t(CB), B0 - off));
    mbar_arrive_expect_tx(&full[st], bytes);
    bulk_load(ring + size_t(st) * CB, dbytes + off, bytes, &full[st]);
  };
  if constexpr (RING) {
    if (threadIdx.x == 0) {
      for (uint32_t i = 0; i < NST; ++i) mbar_init(&full[i], 1);
      *abort = 0;
      fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0)
      while (issued < nchunks && issued < int64_t(NST)) issue(issued++);
  }
  griddep_wait();  // outputs cleared by the launch before this one (when it is its dependent)
  for (int64_t t = t_begin; t < t_end; ++t) {
    const int64_t w = GAIN ? qt.at(t, 0, p.W, 0) : 0;
    if (GAIN && p.quality) qual_window(p, qa, w, lane);
    const int64_t s0 = t * RS8;  // the step's first byte
    bool have = true;
    if constexpr (RING) {
      const int64_t s1 = min(s0 + RS8, B0);
      if (s1 > s0)
        for (int64_t c = (s0 - A0) >> cshift; c <= (s1 - 1 - A0) >> cshift; ++c)
          have &= mbar_wait_bounded(&full[static_cast<uint32_t>(c) & (NST - 1)],
                                    static_cast<uint32_t>(c >> ceil_log2(NST)) & 1u, abort);
    }
    // one rank row's durations: from the ring when the whole row lies below
    // B0 (ring offsets wrap), else from global memory
    auto in_ring = [&](int64_t r) { return RING && s0 + (r + 1) * S * 8 <= B0; };
    auto ring_off = [&](int64_t r) { return static_cast<uint32_t>(s0 + r * S * 8 - A0) & RBmask; };
    int64_t b0[SMAX], b1[SMAX];
    int32_t br[SMAX];
    uint64_t slow = 0;
#pragma unroll
    for (int s = 0; s < SMAX; ++s) {
      b0[s] = BASE ? 0 : -1;
      b1[s] = 0;
      br[s] = 0;
    }
    if constexpr (!VEC) {
      // one rank row at a time per thread, in increasing rank order (a strict
      // '>' keeps the lowest rank), each duration loaded where it is used
      for (int64_t r = threadIdx.x; r < R; r += kGenThreads) {
        const int64_t* row = d + (t * R + r) * S;
        const bool rr = in_ring(r);
        const uint32_t ro = RING ? ring_off(r) : 0u;
        auto val = [&](int s) -> int64_t {
          if (RING && rr) return *reinterpret_cast<const int64_t*>(ring + ((ro + 8u * s) & RBmask));
          return __ldg(row + s);
        };
        int64_t P = 0, other = 0;
#pragma unroll
        for (int s = 0; s < SMAX; ++s) {
          if (s >= S) break;
          const int64_t v = have ? val(s) : 0;
          dor |= hi32(v);
          P += v;
          if (s == p.other_stage) other = v;
          if (BASE) {
            b0[s] = v > b0[s] ? v : b0[s];
            b1[s] += v;
          } else if (P > b0[s]) {
            b0[s] = P;
            br[s] = static_cast<int32_t>(r);
          }
        }
        tor |= hi32(P);
        if (BASE) {
          const uint64_t k = (static_cast<uint64_t>(P) << 16) | static_cast<uint64_t>(65535 - r);
          slow = k > slow ? k : slow;
        }
        if (GAIN) {
          const int64_t* mr = p.m + (w * R + r) * S;
#pragma unroll
          for (int s = 0; s < SMAX; ++s) {
            if (s >= S) break;
            int64_t cut = (have ? val(s) : 0) - __ldg(mr + s);
            cut = cut > 0 ? cut : 0;
            b1[s] = (P - cut) > b1[s] ? (P - cut) : b1[s];
          }
          if (p.quality) qual_row(p, qa, t, r, P, other, dor);
        }
      }
    } else {
      // even S (frontier and baseline passes): rows start 16-byte aligned and
      // are loaded whole with 16-byte loads, one row in flight per thread
      static_assert(!GAIN, "the evidence pass loads durations where it uses them");
      for (int64_t r = threadIdx.x; r < R; r += kGenThreads) {
        const int64_t* row = d + (t * R + r) * S;
        const bool rr = in_ring(r);
        const uint32_t ro = RING ? ring_off(r) : 0u;
        int64_t v[SMAX];
#pragma unroll
        for (int s = 0; s < SMAX; s += 2) {
          if (s >= S) break;
          longlong2 x = make_longlong2(0, 0);
          if (RING && rr) {
            if (have) x = *reinterpret_cast<const longlong2*>(ring + ((ro + 8u * s) & RBmask));
          } else {
            x = __ldg(reinterpret_cast<const longlong2*>(row + s));
          }
          v[s] = x.x;
          v[s + 1] = x.y;
        }
        int64_t P = 0;
#pragma unroll
        for (int s = 0; s < SMAX; ++s) {
          if (s >= S) break;
          dor |= hi32(v[s]);
          P += v[s];
          if (BASE) {
            b0[s] = v[s] > b0[s] ? v[s] : b0[s];
            b1[s] += v[s];
          } else if (P > b0[s]) {
            b0[s] = P;
            br[s] = static_cast<int32_t>(r);
          }
        }
        tor |= hi32(P);
        if (BASE) {
          const uint64_t k = (static_cast<uint64_t>(P) << 16) | static_cast<uint64_t>(65535 - r);
          slow = k > slow ? k : slow;
        }
      }
    }
#pragma unroll
    for (int s = 0; s < SMAX; ++s) {
      if (s >= S) break;
      uint64_t k0;
      if (BASE) k0 = static_cast<uint64_t>(b0[s]);
      else k0 = b0[s] < 0 ? 0ull : (static_cast<uint64_t>(b0[s]) << 16) | static_cast<uint64_t>(65535 - br[s]);
      const uint64_t m0 = warp_max_u64(k0);
      const uint64_t m1 = GAIN   ? warp_max_u64(static_cast<uint64_t>(b1[s]))
                          : BASE ? warp_sum_u64(static_cast<uint64_t>(b1[s]))
                                 : 0;
      if (lane == 0) {
        red[warp][s] = m0;
        red[warp][32 + s] = m1;
      }
    }
    if (BASE) {
      const uint64_t ks = warp_max_u64(slow);
      if (lane == 0) red[warp][64] = ks;
    }
    __syncthreads();
    if (warp == 0) {
      uint64_t v0 = 0, v1 = 0, v2 = 0;
      if (lane < S)
        for (int ww = 0; ww < kGenThreads / 32; ++ww) {
          v0 = red[ww][lane] > v0 ? red[ww][lane] : v0;
          if (BASE) v1 += red[ww][32 + lane];
          else v1 = red[ww][32 + lane] > v1 ? red[ww][32 + lane] : v1;
        }
      if (BASE)
        for (int ww = 0; ww < kGenThreads / 32; ++ww) v2 = red[ww][64] > v2 ? red[ww][64] : v2;
      if (GAIN) finalize_gain(p, S, t, v0, static_cast<int64_t>(v1), lane, acc);
      else if (BASE) finalize_base(p, S, t, v0, v1, v2, lane, bacc);
      else finalize_frontier(p, S, t, v0, lane, acc);
    }
    __syncthreads();
    if constexpr (RING) {
      // every thread is done with step t: the chunks wholly before the next
      // step's first byte are free, and each freed stage takes the next chunk
      if (threadIdx.x == 0) {
        const int64_t free_upto = min(nchunks, (s0 + RS8 - A0) >> cshift);
        if (released < free_upto && issued < nchunks) fence_proxy_async_smem();
        for (; released < free_upto; ++released)
          if (issued < nchunks) issue(issued++);
      }
    }
  }
  if constexpr (RING) {
    // copies still in flight (only when a wait gave up): let them land before
    // the CTA's shared memory is released
    if (threadIdx.x == 0)
      for (int64_t c = released; c < issued; ++c)
        mbar_wait_timeout(&full[static_cast<uint32_t>(c) & (NST - 1)], static_cast<uint32_t>(c >> ceil_log2(NST)) & 1u);
  }
  if (BASE && warp == 0) flush_base(p, S, bacc, lane);
  if (!BASE && p.X && warp == 0) flush_window(p, S, acc, lane);
  if (GAIN && p.quality) qual_window(p, qa, -2, lane);
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), __reduce_or_sync(kFull, tor)) |
                        ((RING && *abort) ? SF_ST_TIMEOUT : 0u);
  if (lane == 0) report(p.status, bits);
}

// Warp-per-step generic path (S <= 16, many steps): each warp takes every
// eighth step of its CTA's range alone (rank rows lane, lane + 32, ... in
// increasing order, so a strict '>' keeps the lowest rank), reduces the
// stages with warp reductions and runs the step's epilogue itself, with its
// own window accumulators: no CTA barrier, eight independent steps in flight
// per CTA.  (The CTA-per-step kernel above spends about 5 us per step behind
// two barriers.)
template <int SMAX, int MODE, bool VEC>
__global__ void __launch_bounds__(kGenThreads)
    stream_warp_kernel(const int64_t* __restrict__ d, const Params p) {
  constexpr bool GAIN = MODE == 1;
  constexpr bool BASE = MODE == 2;
  constexpr int UG = SMAX > 8 ? 1 : 2;  // rank rows in flight per lane (frontier, baselines)
  constexpr int kWarps = kGenThreads / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = static_cast<int>(p.S);
  const int64_t R = p.R;
  const int64_t NB = gridDim.x, b = blockIdx.x;
  const int64_t t_begin = p.T * b / NB, t_end = p.T * (b + 1) / NB;
  uint32_t dor = 0, tor = 0;
  WinAcc acc;
  QualAcc qa;
  WinTrack qt;  // window of the warp's step (evidence pass)
  BaseAcc bacc;
  griddep_wait();  // outputs cleared by the launch before this one (when it is its dependent)
  for (int64_t t = t_begin + warp; t < t_end; t += kWarps) {
    const int64_t w = GAIN ? qt.at(t, 0, p.W, 0) : 0;
    if (GAIN && p.quality) qual_window(p, qa, w, lane);
    int64_t b0[SMAX], b1[SMAX];
    int32_t br[SMAX];
    uint64_t slow = 0;
#pragma unroll
    for (int s = 0; s < SMAX; ++s) {
      b0[s] = BASE ? 0 : -1;
      b1[s] = 0;
      br[s] = 0;
    }
    if constexpr (GAIN) {
      // evidence pass: one row at a time, durations loaded where used
      for (int64_t r = lane; r < R; r += 32) {
        const int64_t* row = d + (t * R + r) * S;
        int64_t P = 0, other = 0;
#pragma unroll
        for (int s = 0; s < SMAX; ++s) {
          if (s >= S) break;
          const int64_t v = __ldg(row + s);
          dor |= hi32(v);
          P += v;
          if (s == p.other_stage) other = v;
          if (P > b0[s]) {
            b0[s] = P;
            br[s] = static_cast<int32_t>(r);
          }
        }
        tor |= hi32(P);
        const int64_t* mr = p.m + (w * R + r) * S;
#pragma unroll
        for (int s = 0; s < SMAX; ++s) {
          if (s >= S) break;
          int64_t cut = __ldg(row + s) - __ldg(mr + s);
          cut = cut > 0 ? cut : 0;
          b1[s] = (P - cut) > b1[s] ? (P - cut) : b1[s];
        }
        if (p.quality) qual_row(p, qa, t, r, P, other, dor);
      }
    } else {
      for (int64_t r0 = lane; r0 < R; r0 += 32 * UG) {
        int64_t v[UG][SMAX];
#pragma unroll
        for (int u = 0; u < UG; ++u) {
          const int64_t r = r0 + 32 * u;
          if (r >= R) break;
          const int64_t* row = d + (t * R + r) * S;
          if constexpr (VEC) {  // S even: rows start 16-byte aligned
#pragma unroll
            for (int s = 0; s < SMAX; s += 2) {
              if (s >= S) break;
              const longlong2 x = __ldg(reinterpret_cast<const longlong2*>(row + s));
              v[u][s] = x.x;
              v[u][s + 1] = x.y;
            }
          } else {
#pragma unroll
            for (int s = 0; s < SMAX; ++s) {
              if (s >= S) break;
              v[u][s] = __ldg(row + s);
            }
          }
        }
#pragma unroll
        for (int u = 0; u < UG; ++u) {
          const int64_t r = r0 + 32 * u;
          if (r >= R) break;
          int64_t P = 0;
#pragma unroll
          for (int s = 0; s < SMAX; ++s) {
            if (s >= S) break;
            dor |= hi32(v[u][s]);
            P += v[u][s];
            if (BASE) {
              b0[s] = v[u][s] > b0[s] ? v[u][s] : b0[s];
              b1[s] += v[u][s];
            } else if (P > b0[s]) {
              b0[s] = P;
              br[s] = static_cast<int32_t>(r);
            }
          }
          tor |= hi32(P);
          if (BASE) {
            const uint64_t k = (static_cast<uint64_t>(P) << 16) | static_cast<uint64_t>(65535 - r);
            slow = k > slow ? k : slow;
          }
        }
      }
    }
    // lane s keeps stage s's reductions
    uint64_t v0 = 0, v1 = 0;
#pragma unroll
    for (int s = 0; s < SMAX; ++s) {
      if (s >= S) break;
      uint64_t k0;
      if (BASE) k0 = static_cast<uint64_t>(b0[s]);
      else k0 = b0[s] < 0 ? 0ull : (static_cast<uint64_t>(b0[s]) << 16) | static_cast<uint64_t>(65535 - br[s]);
      const uint64_t m0 = warp_max_u64(k0);
      const uint64_t m1 = GAIN   ? warp_max_u64(static_cast<uint64_t>(b1[s]))
                          : BASE ? warp_sum_u64(static_cast<uint64_t>(b1[s]))
                                 : 0;
      if (lane == s) {
        v0 = m0;
        v1 = m1;
      }
    }
    if (GAIN) finalize_gain(p, S, t, v0, static_cast<int64_t>(v1), lane, acc);
    else if (BASE) finalize_base(p, S, t, v0, v1, warp_max_u64(slow), lane, bacc);
    else finalize_frontier(p, S, t, v0, lane, acc);
  }
  if (BASE) flush_base(p, S, bacc, lane);
  if (!BASE && p.X) flush_window(p, S, acc, lane);
  if (GAIN && p.quality) qual_window(p, qa, -2, lane);
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), __reduce_or_sync(kFull, tor));
  if (lane == 0) report(p.status, bits);
}

// --------------------------------------------------------------------------
// Host side

// Launch `kern` on `stream`; with `pdl`, as the programmatic dependent of the
// previous launch on the stream (this call's clear of its outputs: the kernel
// streams its first tiles while the clear runs and writes after griddep_wait).
template <typename... KArgs, typename... Args>
cudaError_t launch_ex(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream, bool pdl,
                      Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

template <int S, int MODE>
cudaError_t prepare_fast() {
  return cudaFuncSetAttribute(stream_kernel<S, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(kSmemBytes));
}

template <int MODE>
cudaError_t dispatch_fast(int S, const CUtensorMap& map, const CUtensorMap& map_m, const Params& p, int grid,
                          cudaStream_t stream, bool pdl) {
#define SF_CASE(SV)                                                                                    \
  case SV: {                                                                                           \
    cudaError_t e = prepare_fast<SV, MODE>();                                                          \
    if (e != cudaSuccess) return e;                                                                    \
    return launch_ex(stream_kernel<SV, MODE>, grid, kBlockThreads, kSmemBytes, stream, pdl, map, map_m, p); \
  }
  switch (S) {
    SF_CASE(2)
    SF_CASE(4)
    SF_CASE(6)
    SF_CASE(8)
    SF_CASE(10)
    SF_CASE(12)
    SF_CASE(14)
    SF_CASE(16)
    default:
      return cudaErrorInvalidValue;
  }
#undef SF_CASE
}

cudaError_t dispatch_lanes(int S, int G, const CUtensorMap& map, const Params& p, int grid, cudaStream_t stream,
                           bool pdl) {
#define SF_LANES(SV, GV)                                                                          \
  if (S == SV && G == GV) {                                                                       \
    cudaError_t e = cudaFuncSetAttribute(lanes_kernel<SV, GV>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                                         static_cast<int>(kSmemBytes));                          \
    if (e != cudaSuccess) return e;                                                               \
    return launch_ex(lanes_kernel<SV, GV>, grid, kBlockThreads, kSmemBytes, stream, pdl, map, p);   \
  }
  SF_LANES(2, 2)
  SF_LANES(2, 4)
  SF_LANES(2, 8)
  SF_LANES(4, 2)
  SF_LANES(4, 4)
  SF_LANES(4, 8)
  SF_LANES(8, 2)
  SF_LANES(8, 4)
  SF_LANES(16, 2)
#undef SF_LANES
  return cudaErrorInvalidValue;
}

}  // namespace

EncodeFn encode_fn() {
  static EncodeFn fn = [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      f = nullptr;
    return reinterpret_cast<EncodeFn>(f);
  }();
  return fn;
}

cudaError_t launch_stream_pass(const StreamJob& j, cudaStream_t stream) {
  Params p{};
  p.T = j.T;
  p.R = j.R;
  p.S = j.S;
  p.a = j.a;
  p.lead = j.lead;
  p.mk = j.mk;
  p.X = j.X;
  p.D = j.D;
  p.E = j.E;
  p.C = j.C;
  p.step_lead = j.step_lead;
  p.t0 = j.t0;
  p.W = j.W;
  p.w_first = j.t0 / j.W;
  p.m = j.m;
  p.wall = j.wall;
  p.other_stage = j.other_stage;
  p.eta_num = j.eta_num;
  p.eta_den = j.eta_den;
  p.Y = j.Y;
  p.quality = j.quality;
  p.status = j.status;
  p.d = j.d;
  p.bM = j.bM;
  p.bSUM = j.bSUM;
  p.bSLOW = j.bSLOW;
  p.bRANK0 = j.bRANK0;

  const int64_t RS = j.R * j.S;
  const int64_t step_rows = RS / 16;
  const int64_t rows_total = j.T * step_rows;
  const bool fast = (j.S % 2 == 0) && j.S <= 16 && (RS % 16 == 0) &&
                    rows_total <= int64_t(0x7fffffff) && encode_fn() != nullptr &&
                    (reinterpret_cast<uintptr_t>(j.d) % 16 == 0) &&
                    (!j.gain || reinterpret_cast<uintptr_t>(j.m) % 16 == 0);
  const int sms = sm_count();
  // fewer steps than SMs over many ranks (frontier and aggregation): split
  // each step's ranks over a cluster so that every SM streams
  if (!j.gain && !j.base && j.T < sms && j.R >= 1024 && (j.S % 2 == 0) && j.S <= 16 &&
      reinterpret_cast<uintptr_t>(j.d) % 16 == 0) {
    const int csize = split_cluster(static_cast<int>(j.S), j.T, j.R);
    count_launch();
    cudaError_t e = dispatch_split(static_cast<int>(j.S), j.d, p, csize, stream, j.after_clear);
    if (e != cudaSuccess && csize > 8) {  // a 16-CTA cluster that cannot be placed: portable size
      cudaGetLastError();
      e = dispatch_split(static_cast<int>(j.S), j.d, p, 8, stream, j.after_clear);
    }
    return e;
  }
  if (fast) {
    p.step_rows = step_rows;
    // frontier and aggregation over small steps: several steps per warp instruction
    const int lanes = (!j.gain && !j.base) ? lanes_groups(j.R, j.S) : 0;
    if (step_rows <= kR0MaxRows) {
      p.regime = 0;
      p.K = static_cast<int>(kR0MaxRows / step_rows);
      if (lanes > 0) p.K = lanes * static_cast<int>(kR0MaxRows / (lanes * step_rows));  // whole rounds of G steps
      p.box_rows = static_cast<int>(p.K * step_rows);
      p.tiles_per_step = 0;
    } else {
      p.regime = 1;
      // rows per rank-aligned block: a tile must hold whole rank rows
      const int64_t elems = 16 * j.S / std::gcd<int64_t>(16, j.S);  // lcm(16, S)
      const int64_t q = elems / 16;
      const int64_t max_rows = j.gain ? kR1GainMaxRows : kR1MaxRows;
      int64_t n = (step_rows + max_rows - 1) / max_rows, br = 0;
      for (;; ++n) {
        br = (step_rows + n - 1) / n;
        br = (br + q - 1) / q * q;
        if (br <= max_rows) break;
      }
      p.box_rows = static_cast<int>(br);
      p.tiles_per_step = static_cast<int>((step_rows + br - 1) / br);
      p.K = 0;
    }
    // the small-step frontier pass reads every shape it takes (S = 2 too) 128B-swizzled
    const bool swz = (j.S == 4 || j.S == 8 || j.S == 16) || lanes > 0;
    auto encode = [&](CUtensorMap* out, const int64_t* base, int64_t rows) {
      const cuuint64_t gdim[2] = {16, static_cast<cuuint64_t>(rows)};
      const cuuint64_t gstride[1] = {kRowBytes};
      const cuuint32_t box[2] = {16, static_cast<cuuint32_t>(p.box_rows)};
      const cuuint32_t estride[2] = {1, 1};
      return encode_fn()(out, CU_TENSOR_MAP_DATA_TYPE_INT64, 2, const_cast<int64_t*>(base), gdim, gstride, box,
                         estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                         swz ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    };
    CUtensorMap map, map_m;
    if (encode(&map, j.d, rows_total) != CUDA_SUCCESS) return cudaErrorInvalidValue;
    map_m = map;
    p.m_by_tma = (j.gain && p.regime == 1) ? 1 : 0;
    p.nst = p.regime == 0 ? kR0Stages : p.m_by_tma ? kR1GainStages : kR1Stages;
    p.stage_bytes = p.regime == 0 ? kR0StageBytes : p.m_by_tma ? kR1GainStageBytes : kR1StageBytes;
    // Small steps in regime 1: groups of warps take steps in turn, so that
    // several steps' reductions are in flight.  Each group owns nst / groups
    // ring stages: a stage is refilled only after its own group has consumed
    // it, so no wait can pass a phase early.
    p.groups = 1;
    if (p.regime == 1 && p.nst >= 4) p.groups = p.tiles_per_step == 1 && step_rows <= 128 ? 4 : p.tiles_per_step <= 2 ? 2 : 1;
    if (p.m_by_tma) {
      const int64_t nW = (j.T + j.W - 1) / j.W;
      if (nW * step_rows > int64_t(0x7fffffff) || encode(&map_m, j.m, nW * step_rows) != CUDA_SUCCESS)
        return cudaErrorInvalidValue;
    }
    const int64_t units = p.regime == 0 ? (j.T + p.K - 1) / p.K : j.T;
    const int grid = static_cast<int>(std::min<int64_t>(sms, units));
    count_launch();
    const bool pdl = j.after_clear;
    if (lanes > 0) return dispatch_lanes(static_cast<int>(j.S), lanes, map, p, grid, stream, pdl);
    if (j.base) return dispatch_fast<2>(static_cast<int>(j.S), map, map_m, p, grid, stream, pdl);
    return j.gain ? dispatch_fast<1>(static_cast<int>(j.S), map, map_m, p, grid, stream, pdl)
                  : dispatch_fast<0>(static_cast<int>(j.S), map, map_m, p, grid, stream, pdl);
  }
  count_launch();
  const bool vec = j.S % 2 == 0;  // whole-row 16-byte loads (frontier and baseline passes)
  // bulk-copy ring: the smallest power-of-two chunk (4-16 KB) of which
  // kGenRingStages - 1 hold a whole step; larger steps read global memory
  const int64_t step_bytes = j.R * j.S * 8;
  uint32_t chunk = 0;
  for (uint32_t c = 4096; c <= 16384 && !chunk; c *= 2)
    if (step_bytes <= int64_t(kGenRingStages - 1) * c) chunk = c;
  p.stage_bytes = static_cast<int>(chunk);
  p.nst = static_cast<int>(kGenRingStages);
  auto generic = [&](auto smax) {
    constexpr int SM = decltype(smax)::value;
    const bool pdl = j.after_clear;
    auto go = [&](auto kern, bool ring) {
      const size_t smem = ring ? size_t(kGenRingStages) * chunk : 0;
      int per_sm = 4;
      if (ring) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kGenThreads, smem);
        if (e != cudaSuccess) return e;
        per_sm = std::max(per_sm, 1);
      }
      const int grid = static_cast<int>(std::min<int64_t>(int64_t(sms) * per_sm, j.T));
      return launch_ex(kern, grid, kGenThreads, smem, stream, pdl, j.d, p);
    };
    if constexpr (SM > 16) {
      // more than 16 stages: registers hold these kernels to one or two CTAs
      // per SM, and the bulk-copy ring keeps the loads off their step chain
      // (512 x 24: 0.434 -> 0.405 ms).  Up to 16 stages four CTAs per SM
      // hide the loads better than a ring that leaves room for three (1000 x 5:
      // 0.229 against 0.285 ms), so those shapes read global memory.
      if (chunk != 0) {
        if (j.gain) return go(stream_generic_kernel<SM, 1, false, true>, true);
        if (j.base && vec) return go(stream_generic_kernel<SM, 2, true, true>, true);
        if (j.base) return go(stream_generic_kernel<SM, 2, false, true>, true);
        if (vec) return go(stream_generic_kernel<SM, 0, true, true>, true);
        return go(stream_generic_kernel<SM, 0, false, true>, true);
      }
    }
    if constexpr (SM <= 16) {
      // many steps: one warp per step (see stream_warp_kernel); few steps
      // keep a CTA per step so that a step's ranks still spread over 256 threads
      if (j.T >= int64_t(sms) * 4 * (kGenThreads / 32)) {
        auto gow = [&](auto kern) {
          int per_sm = 1;
          cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kGenThreads, 0);
          if (e != cudaSuccess) return e;
          const int grid = static_cast<int>(std::min<int64_t>(int64_t(sms) * std::max(per_sm, 1),
                                                              (j.T + kGenThreads / 32 - 1) / (kGenThreads / 32)));
          return launch_ex(kern, grid, kGenThreads, 0, stream, pdl, j.d, p);
        };
        if (j.gain) return gow(stream_warp_kernel<SM, 1, false>);
        if (j.base && vec) return gow(stream_warp_kernel<SM, 2, true>);
        if (j.base) return gow(stream_warp_kernel<SM, 2, false>);
        if (vec) return gow(stream_warp_kernel<SM, 0, true>);
        return gow(stream_warp_kernel<SM, 0, false>);
      }
    }
    if (j.gain) return go(stream_generic_kernel<SM, 1, false, false>, false);
    if (j.base && vec) return go(stream_generic_kernel<SM, 2, true, false>, false);
    if (j.base) return go(stream_generic_kernel<SM, 2, false, false>, false);
    if (vec) return go(stream_generic_kernel<SM, 0, true, false>, false);
    return go(stream_generic_kernel<SM, 0, false, false>, false);
  };
  if (j.S <= 4) return generic(std::integral_constant<int, 4>{});
  if (j.S <= 8) return generic(std::integral_constant<int, 8>{});
  if (j.S <= 16) return generic(std::integral_constant<int, 16>{});
  return generic(std::integral_constant<int, 32>{});
}

}  // namespace sf

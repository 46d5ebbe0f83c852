// sf_select.cu - the per-window kernels of libstagefrontier:
//   * window_median: lower median of every (window, rank, stage) column
//     (the per-rank window baseline of Sec. 4, Eq. 4);
//   * topk: top-k stages by X and (stage, rank) pairs by lead-rank credit E;
//   * gates: App. C label gates, routing and ambiguity sets, fp64 shares/gains;
//   * zero: clears accumulators the library owns the semantics of.
#include <algorithm>

#include <cooperative_groups.h>

#include "sf_device.cuh"
#include "sf_launch.h"

namespace sf {

namespace {

__device__ __forceinline__ int64_t imin64(int64_t a, int64_t b) { return a < b ? a : b; }

__global__ void zero_kernel(uint32_t* __restrict__ p, size_t words) {
  for (size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x; i < words;
       i += size_t(gridDim.x) * blockDim.x)
    p[i] = 0u;
}

// ---------------------------------------------------------------------------
// Lower median, one warp per column.  A CTA of 8 warps owns (window w, eight
// consecutive flat columns c = r*S + s).  The window's rows of those columns
// are read coalesced and transposed through shared memory so each warp holds
// its column in registers (NPL values per lane).  Values are mapped to an
// order-preserving unsigned key (so any int64 input is handled exactly) and
// offset by the column minimum; the k-th smallest offset (k = floor((n-1)/2))
// is then found by radix selection, most significant 8-bit digit first: a
// per-warp 256-bin shared-memory histogram of the digit among the values that
// share the digits chosen so far, a warp scan to find the bin holding rank k,
// and the rank re-based into that bin.  A 24-bit spread takes three passes.
constexpr int kMedCols = 8;
constexpr int kMedThreads = kMedCols * 32;
constexpr int kMedBins = 256;
// Per-warp counters: 256 digit bins, then 32 per-lane discard slots that
// non-matching and padding values increment instead of branching around the
// atomic.  288 words = 1152 bytes keeps every warp's block 16-byte aligned.
constexpr int kMedHistWords = kMedBins + 32;

// k-th smallest (0-based) of the lane-strided values get(i) (row lane + 32 i,
// valid while row < n), all below 2^nbits.  hist: this warp's 256 counters.
template <typename U, int NPL, typename Get>
__device__ __forceinline__ U warp_radix_select(Get get, int n, int nbits, uint32_t k, uint32_t* hist,
                                               int lane) {
  U prefix = 0;
  int shift = nbits;
  uint32_t rem = k;
  bool first = true;
  while (shift > 0) {
    const int D = shift < 8 ? shift : 8;
    shift -= D;
    const uint32_t dmask = (1u << D) - 1u;
    const int hs = shift + D;  // bits above the current digit
    reinterpret_cast<uint4*>(hist)[2 * lane] = make_uint4(0, 0, 0, 0);
    reinterpret_cast<uint4*>(hist)[2 * lane + 1] = make_uint4(0, 0, 0, 0);
    __syncwarp();
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
      if (lane + 32 * i < n) {
        const U v = get(i);
        if (first || (v >> hs) == prefix)
          atomicAdd(&hist[static_cast<uint32_t>(v >> shift) & dmask], 1u);
      }
    }
    __syncwarp();
    const uint4 h0 = reinterpret_cast<const uint4*>(hist)[2 * lane];
    const uint4 h1 = reinterpret_cast<const uint4*>(hist)[2 * lane + 1];
    const uint32_t hb[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
    uint32_t sum = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) sum += hb[j];
    uint32_t incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t up = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += up;
    }
    const uint32_t excl = incl - sum;
    const int owner = __ffs(__ballot_sync(kFull, excl <= rem && rem < incl)) - 1;
    uint32_t digit = 0, below = excl;
    if (lane == owner) {
      uint32_t c = excl;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (rem >= c && rem < c + hb[j]) {
          digit = 8u * lane + j;
          below = c;
        }
        c += hb[j];
      }
    }
    digit = __shfl_sync(kFull, digit, owner);
    below = __shfl_sync(kFull, below, owner);
    rem -= below;
    prefix = (prefix << D) | static_cast<U>(digit);
    first = false;
    __syncwarp();
  }
  return prefix;
}

// Shared-memory increment of one counter, issued only when `pred` is set
// (explicitly predicated, so a warp never branches around it).
__device__ __forceinline__ void red_shared_inc_if(uint32_t* counter, bool pred) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.u32 p, %1, 0;\n\t@p red.shared.add.u32 [%0], 1;\n\t}" ::"r"(smem_u32(counter)),
      "r"(static_cast<uint32_t>(pred))
      : "memory");
}

// The k-th smallest of the live values among x[i] (row lane + 32 i), all
// below 2^nbits.  Padding slots must hold 2^nbits - 1: they sort at or after
// every live value, so counting them never moves the rank-k bin and no slot
// needs a validity test.  The first digit takes the top 8 bits of the range,
// [nbits - 8, nbits), so it spreads over the 256 bins and its chosen bin
// usually holds a few percent of the column; the next pass then keeps the
// values of that bin as candidates (in this warp's own, already consumed
// column slots of the tile: slot j at cand(j)) and every later pass reads only
// those; a bin of at most 32 values is finished directly, one value per lane,
// by counting.  A bin too full to keep (heavy ties) falls back to predicated
// increments over all slots.
template <int NPL, typename CandAddr>
__device__ __forceinline__ uint32_t warp_select_bits32(const uint32_t (&x)[NPL], int nbits, uint32_t k,
                                                       uint32_t* hist, int lane, CandAddr cand) {
  constexpr uint32_t kCap = 32u * NPL < 512u ? 32u * NPL : 512u;  // candidate slots
  if (nbits == 0) return 0;
  int sh = nbits > 8 ? nbits - 8 : 0;
  reinterpret_cast<uint4*>(hist)[2 * lane] = make_uint4(0, 0, 0, 0);
  reinterpret_cast<uint4*>(hist)[2 * lane + 1] = make_uint4(0, 0, 0, 0);
  __syncwarp();
#pragma unroll
  for (int i = 0; i < NPL; ++i) atomicAdd(&hist[x[i] >> sh], 1u);  // x < 2^nbits: the bin is below 256
  __syncwarp();
  uint32_t digit, below;
  hist_find(hist, k, lane, digit, below);
  uint32_t rem = k - below;
  uint32_t prefix = digit << sh;
  const uint32_t kept = hist[digit];  // values the next pass matches
  int hi = sh;                        // offset bits at and above hi are chosen
  if (hi == 0) return prefix;
  uint32_t* ncand = hist + 256;  // spare word after the bins
  if (kept <= 32) {
    // at most one value of the chosen bin per lane: gather them, sort the
    // warp's 32 values with a bitonic network (lanes past the bin hold the
    // largest key, which sorts last) and take the rem-th smallest, instead
    // of more histogram passes
    __syncwarp();
    if (lane == 0) *ncand = 0;
    __syncwarp();
#pragma unroll
    for (int i = 0; i < NPL; ++i)
      if ((x[i] >> hi) == digit) *cand(atomicAdd(ncand, 1u)) = x[i];
    __syncwarp();
    uint32_t v = static_cast<uint32_t>(lane) < kept ? *cand(lane) : 0xffffffffu;
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
      for (int stride = size >> 1; stride > 0; stride >>= 1) {
        const uint32_t o = __shfl_xor_sync(kFull, v, stride);
        // ascending within blocks whose `size` bit is clear; the lower lane of a pair keeps the smaller
        const bool up = (lane & size) == 0, low = (lane & stride) == 0;
        v = (up == low) ? min(v, o) : max(v, o);
      }
    }
    const uint32_t ans = __shfl_sync(kFull, v, static_cast<int>(rem));
    __syncwarp();
    return ans;
  }
  const bool compact = kept <= kCap;
  bool keep_pass = compact;  // the next pass keeps the candidates
  __syncwarp();
  while (hi > 0) {
    sh = hi > 8 ? hi - 8 : 0;
    const uint32_t mask = (1u << (hi - sh)) - 1u;
    reinterpret_cast<uint4*>(hist)[2 * lane] = make_uint4(0, 0, 0, 0);
    reinterpret_cast<uint4*>(hist)[2 * lane + 1] = make_uint4(0, 0, 0, 0);
    if (lane == 0) *ncand = 0;
    __syncwarp();
    if (!compact) {
#pragma unroll
      for (int i = 0; i < NPL; ++i)
        red_shared_inc_if(&hist[(x[i] >> sh) & mask], (x[i] >> hi) == (prefix >> hi));
    } else if (keep_pass) {
      // the pass after the first: count and keep the matching values
#pragma unroll
      for (int i = 0; i < NPL; ++i) {
        if ((x[i] >> hi) == (prefix >> hi)) {
          atomicAdd(&hist[(x[i] >> sh) & mask], 1u);
          *cand(atomicAdd(ncand, 1u)) = x[i];
        }
      }
    } else {
      for (uint32_t j = lane; j < kept; j += 32) {
        const uint32_t v = *cand(j);
        red_shared_inc_if(&hist[(v >> sh) & mask], (v >> hi) == (prefix >> hi));
      }
    }
    __syncwarp();
    hist_find(hist, rem, lane, digit, below);
    rem -= below;
    prefix |= digit << sh;
    hi = sh;
    keep_pass = false;
    __syncwarp();
  }
  return prefix;
}

template <int NPL, bool kVec>
__global__ void __launch_bounds__(kMedThreads)
    median_kernel(const int64_t* __restrict__ d, int64_t T, int64_t RS, int64_t W, int64_t ngroups,
                  int64_t* __restrict__ m) {
  constexpr int LD = 32 * NPL + 1;
  extern __shared__ int64_t colbuf[];  // [kMedCols][LD], then kMedCols x 256 histogram counters
  // kMedCols * LD * 8 bytes is a multiple of 64, so the counters start 16-byte aligned
  uint32_t* hists = reinterpret_cast<uint32_t*>(colbuf + kMedCols * LD);
  const int64_t w = blockIdx.x / ngroups;
  const int64_t c0 = (blockIdx.x % ngroups) * kMedCols;
  const int ncols = static_cast<int>(imin64(kMedCols, RS - c0));
  const int64_t tb = w * W;
  const int n = static_cast<int>(imin64(W, T - tb));
  const int64_t* base = d + tb * RS + c0;
  if (kVec && ncols == kMedCols) {  // 16-byte loads of column pairs (RS even)
    for (int idx = threadIdx.x; idx < n * (kMedCols / 2); idx += kMedThreads) {
      const int row = idx / (kMedCols / 2), pr = idx % (kMedCols / 2);
      const longlong2 v = __ldg(reinterpret_cast<const longlong2*>(base + int64_t(row) * RS) + pr);
      colbuf[(2 * pr) * LD + row] = v.x;
      colbuf[(2 * pr + 1) * LD + row] = v.y;
    }
  } else {
    for (int idx = threadIdx.x; idx < n * kMedCols; idx += kMedThreads) {
      const int row = idx / kMedCols, c = idx % kMedCols;
      colbuf[c * LD + row] = c < ncols ? __ldg(base + int64_t(row) * RS + c) : 0;
    }
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (warp >= ncols) return;
  uint32_t* hist = hists + warp * kMedBins;  // 1 KB per warp
  constexpr uint64_t kSign = 1ull << 63;
  uint64_t u[NPL];
  uint64_t lo = ~0ull, hi = 0;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const int row = lane + 32 * i;
    u[i] = row < n ? static_cast<uint64_t>(colbuf[warp * LD + row]) ^ kSign : 0;
    if (row < n) {
      lo = u[i] < lo ? u[i] : lo;
      hi = u[i] > hi ? u[i] : hi;
    }
  }
  lo = warp_min_u64(lo);
  hi = warp_max_u64(hi);
  const uint32_t k = static_cast<uint32_t>((n - 1) / 2);
  const uint64_t range = hi - lo;
  const int nbits = range ? 64 - __clzll(static_cast<long long>(range)) : 0;
  uint64_t ans;
  if (nbits <= 32) {
    uint32_t x[NPL];
#pragma unroll
    for (int i = 0; i < NPL; ++i) x[i] = static_cast<uint32_t>(u[i] - lo);  // padding rows never read
    ans = warp_radix_select<uint32_t, NPL>([&](int i) { return x[i]; }, n, nbits, k, hist, lane);
  } else {
#pragma unroll
    for (int i = 0; i < NPL; ++i) u[i] -= lo;
    ans = warp_radix_select<uint64_t, NPL>([&](int i) { return u[i]; }, n, nbits, k, hist, lane);
  }
  if (lane == 0) m[w * RS + c0 + warp] = static_cast<int64_t>((lo + ans) ^ kSign);
}

// The same selection with the window tile brought in by bulk tensor copies: one
// thread issues the whole (window x 8 columns) tile, up to four 2-D boxes of
// 8 int64 x box_rows, all completing on one mbarrier.  The tile stays row-major
// (64-byte rows) with the 64-byte swizzle, so a warp reading one column down
// 32 rows touches 8 distinct 16-byte bank groups per 16 lanes.  Offsets from
// the column minimum stay in registers only when they fit 32 bits; wider
// columns re-read shared memory on every radix pass.  Registers are capped so
// three CTAs share an SM and one CTA's copy overlaps another's selection.
template <int NPL>
__global__ void __launch_bounds__(kMedThreads, 3)
    median_tma_kernel(const __grid_constant__ CUtensorMap map, int64_t T, int64_t RS, int64_t W,
                      int64_t ngroups, int box_rows, int nbox, int tile_rows, int64_t* __restrict__ m,
                      uint32_t* status) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* tile = align_1024(smem_raw);
  const uint32_t tile_bytes = uint32_t(nbox) * uint32_t(box_rows) * 64u;  // bytes the copies write
  uint32_t* hists = reinterpret_cast<uint32_t*>(tile + uint32_t(tile_rows) * 64u);
  uint64_t* bar = reinterpret_cast<uint64_t*>(hists + kMedCols * kMedHistWords);
  volatile int* abort = reinterpret_cast<volatile int*>(bar + 1);
  const int64_t w = blockIdx.x / ngroups;
  const int64_t c0 = (blockIdx.x % ngroups) * kMedCols;
  const int ncols = static_cast<int>(imin64(kMedCols, RS - c0));
  const int64_t tb = w * W;
  const int n = static_cast<int>(imin64(W, T - tb));
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    *abort = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    mbar_arrive_expect_tx(bar, tile_bytes);
    for (int b = 0; b < nbox; ++b)
      tma_load_2d(tile + size_t(b) * box_rows * 64, &map, static_cast<int32_t>(c0),
                  static_cast<int32_t>(tb + int64_t(b) * box_rows), bar);
  }
  const bool ok = mbar_wait_bounded(bar, 0, abort);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (!ok) {
    if (threadIdx.x == 0) {
      report(status, SF_ST_TIMEOUT);
      mbar_wait_timeout(bar, 0);  // let the copies land before the CTA's memory is released
    }
    return;
  }
  if (warp >= ncols) return;
  uint32_t* hist = hists + warp * kMedHistWords;
  // Row lane + 32 i of this warp's column: the 64-byte swizzle term depends
  // only on (row >> 1) & 3 = (lane >> 1) & 3, so each lane has one base and a
  // fixed 2048-byte stride.
  const unsigned char* col = tile + lane * 64 + ((((warp >> 1) ^ ((lane >> 1) & 3)) << 4) | ((warp & 1) << 3));
  // Order-preserving unsigned key of a signed value: flip the sign bit, i.e.
  // bit 31 of the high word.  Most columns share one high word; then the
  // whole selection runs on the 32-bit low words.
  uint32_t xl[NPL];
  const int live = n - lane;  // slot i holds a row of the window iff 32 i < live
  // Low-word min/max over pairs of slots with 3-input min/max; a padding slot
  // repeats row 0's value (row 0 is always in the window) so it cannot move
  // either.  High words only need to agree: OR-accumulate their differences
  // from row 0's high word.
  const uint2 own0 = *reinterpret_cast<const uint2*>(col);  // lane 0's first slot is row 0
  const uint32_t ref_x = __shfl_sync(kFull, own0.x, 0);
  const uint32_t ref_y = __shfl_sync(kFull, own0.y, 0);
  uint32_t lmin = ref_x, lmax = ref_x, hdiff = 0;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const uint2 v = *reinterpret_cast<const uint2*>(col + i * 2048);  // in the tile even for padding slots
    const bool ok = 32 * i < live;
    xl[i] = ok ? v.x : ref_x;
    hdiff |= ok ? (v.y ^ ref_y) : 0u;
  }
#pragma unroll
  for (int i = 0; i + 1 < NPL; i += 2) {
    lmin = __vimin3_u32(lmin, xl[i], xl[i + 1]);
    lmax = __vimax3_u32(lmax, xl[i], xl[i + 1]);
  }
  if (NPL & 1) {
    lmin = min(lmin, xl[NPL - 1]);
    lmax = max(lmax, xl[NPL - 1]);
  }
  const bool narrow = __all_sync(kFull, hdiff == 0);
  const uint32_t hmin = ref_y ^ 0x80000000u, hmax = narrow ? hmin : hmin + 1u;
  const uint32_t k = static_cast<uint32_t>((n - 1) / 2);
  uint64_t key;
  if (hmin == hmax) {
    lmin = __reduce_min_sync(kFull, lmin);
    lmax = __reduce_max_sync(kFull, lmax);
    const uint32_t range = lmax - lmin;
    const int nbits = range ? 32 - __clz(static_cast<int>(range)) : 0;
    const uint32_t pad = nbits == 32 ? 0xffffffffu : (1u << nbits) - 1u;  // sorts at or after every live value
#pragma unroll
    for (int i = 0; i < NPL; ++i) xl[i] = 32 * i < live ? xl[i] - lmin : pad;
    // candidate slot j: this warp's (already consumed) column slot of tile row j
    const uint32_t swz = (warp & 1) << 3;
    auto cand = [&](uint32_t j) {
      return reinterpret_cast<uint32_t*>(tile + j * 64u + ((((warp >> 1) ^ ((j >> 1) & 3u)) << 4) | swz));
    };
    const uint32_t ans = warp_select_bits32<NPL>(xl, nbits, k, hist, lane, cand);
    key = (static_cast<uint64_t>(hmin) << 32) | (lmin + ans);
  } else {
    constexpr uint64_t kSign = 1ull << 63;
    auto ukey = [&](int i) { return static_cast<uint64_t>(*reinterpret_cast<const int64_t*>(col + i * 2048)) ^ kSign; };
    uint64_t lo = ~0ull, hi = 0;
#pragma unroll
    for (int i = 0; i < NPL; ++i)
      if (lane + 32 * i < n) {
        const uint64_t u = ukey(i);
        lo = u < lo ? u : lo;
        hi = u > hi ? u : hi;
      }
    lo = warp_min_u64(lo);
    hi = warp_max_u64(hi);
    const uint64_t range = hi - lo;
    const int nbits = range ? 64 - __clzll(static_cast<long long>(range)) : 0;
    key = lo + warp_radix_select<uint64_t, NPL>([&](int i) { return ukey(i) - lo; }, n, nbits, k, hist, lane);
  }
  if (lane == 0) m[w * RS + c0 + warp] = static_cast<int64_t>(key ^ (1ull << 63));
}

// Windows longer than 1024 steps: the same search, re-reading the column
// from global memory (L2) on every bit.
__global__ void __launch_bounds__(kMedThreads)
    median_global_kernel(const int64_t* __restrict__ d, int64_t T, int64_t RS, int64_t W,
                         int64_t ngroups, int64_t* __restrict__ m) {
  const int64_t w = blockIdx.x / ngroups;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t c = (blockIdx.x % ngroups) * kMedCols + warp;
  if (c >= RS) return;
  const int64_t tb = w * W;
  const int64_t n = imin64(W, T - tb);
  const int64_t* col = d + tb * RS + c;
  constexpr uint64_t kSign = 1ull << 63;
  uint64_t lo = ~0ull, hi = 0;
  for (int64_t t = lane; t < n; t += 32) {
    const uint64_t u = static_cast<uint64_t>(__ldg(col + t * RS)) ^ kSign;
    lo = u < lo ? u : lo;
    hi = u > hi ? u : hi;
  }
  lo = warp_min_u64(lo);
  hi = warp_max_u64(hi);
  const uint64_t k = static_cast<uint64_t>((n - 1) / 2);
  const uint64_t range = hi - lo;
  const int nbits = range ? 64 - __clzll(static_cast<long long>(range)) : 0;
  uint64_t ans = 0;
  for (int bit = nbits - 1; bit >= 0; --bit) {
    const uint64_t cand = ans | (1ull << bit);
    uint32_t cnt = 0;
    for (int64_t t = lane; t < n; t += 32)
      cnt += ((static_cast<uint64_t>(__ldg(col + t * RS)) ^ kSign) - lo) < cand ? 1u : 0u;
    cnt = __reduce_add_sync(kFull, cnt);
    if (cnt <= k) ans = cand;
  }
  if (lane == 0) m[w * RS + c] = static_cast<int64_t>((lo + ans) ^ kSign);
}

// ---------------------------------------------------------------------------
// Top-k.  One CTA per window.  Order: value descending, then index ascending
// (index = stage for X, s*R + r for E); value 0 is not a suspect.
constexpr int kTopThreads = 256;

struct VI {
  int64_t v;
  int64_t i;
};

__device__ __forceinline__ bool before(const VI& a, const VI& b) {  // a ranks ahead of b
  return a.v > b.v || (a.v == b.v && a.i < b.i);
}

__device__ VI block_best(VI x, VI* sm) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    VI y{__shfl_xor_sync(kFull, x.v, o), __shfl_xor_sync(kFull, x.i, o)};
    if (before(y, x)) x = y;
  }
  if (lane == 0) sm[warp] = x;
  __syncthreads();
  VI r = sm[0];
  for (int i = 1; i < kTopThreads / 32; ++i)
    if (before(sm[i], r)) r = sm[i];
  __syncthreads();
  return r;
}

// A window's (stage, rank) entries are split over a cluster of kTopCluster
// CTAs.  Each CTA finds the top k of its slice (k rounds of a block arg-max,
// each round taking the best entry ranked after the previous pick), parks them
// in its shared memory, and the cluster's first CTA merges the cluster's
// k x kTopCluster candidates read through distributed shared memory.
constexpr int kTopCluster = 8;

__global__ void __cluster_dims__(kTopCluster, 1, 1) __launch_bounds__(kTopThreads)
    topk_kernel(const int64_t* __restrict__ X, const int64_t* __restrict__ E, int64_t S, int64_t R, int k,
                int32_t* top_stage, int64_t* top_stage_value, int32_t* top_pair, int64_t* top_pair_value) {
  namespace cg = cooperative_groups;
  cg::cluster_group cluster = cg::this_cluster();
  __shared__ VI sm[kTopThreads / 32];
  __shared__ VI cand[32];
  const unsigned part = cluster.block_rank();
  const int64_t w = blockIdx.x / kTopCluster;
  if (part == 0 && threadIdx.x < 32 && (top_stage || top_stage_value)) {
    const int lane = threadIdx.x;
    const int64_t v = lane < S ? X[w * S + lane] : 0;
    bool taken = false;
    for (int i = 0; i < k; ++i) {
      const uint64_t c = (!taken && lane < S && v > 0) ? static_cast<uint64_t>(v) : 0ull;
      const uint64_t mx = warp_max_u64(c);
      int who = -1;
      if (mx != 0) who = __ffs(__ballot_sync(kFull, c == mx)) - 1;  // lowest stage among equals
      if (lane == who) taken = true;
      if (lane == 0) {
        if (top_stage) top_stage[w * k + i] = who;
        if (top_stage_value) top_stage_value[w * k + i] = who >= 0 ? static_cast<int64_t>(mx) : 0;
      }
    }
  }
  if (E == nullptr || (top_pair == nullptr && top_pair_value == nullptr)) return;  // uniform over the cluster
  const int64_t n = S * R;
  const int64_t chunk = (n + kTopCluster - 1) / kTopCluster;
  const int64_t lo = part * chunk, hi = lo + chunk < n ? lo + chunk : n;
  const int64_t* Ew = E + w * n;
  VI prev{INT64_MAX, -1};
  for (int i = 0; i < k; ++i) {
    VI best{0, INT64_MAX};
    if (prev.v > 0)
      for (int64_t j = lo + threadIdx.x; j < hi; j += kTopThreads) {
        const VI c{Ew[j], j};
        if (c.v > 0 && before(prev, c) && before(c, best)) best = c;  // ranked after the last pick
      }
    best = block_best(best, sm);
    if (threadIdx.x == 0) cand[i] = best;
    prev = best.v > 0 ? best : VI{0, INT64_MAX};
  }
  cluster.sync();
  if (part == 0) {
    const int t = threadIdx.x;
    VI mine{0, INT64_MAX};
    if (t < kTopCluster * k) mine = cluster.map_shared_rank(cand, static_cast<unsigned>(t / k))[t % k];
    prev = VI{INT64_MAX, -1};
    for (int i = 0; i < k; ++i) {
      VI c = (mine.v > 0 && before(prev, mine)) ? mine : VI{0, INT64_MAX};
      c = block_best(c, sm);
      if (threadIdx.x == 0) {
        const bool ok = c.v > 0;
        if (top_pair) {
          top_pair[(w * k + i) * 2 + 0] = ok ? static_cast<int32_t>(c.i / R) : -1;
          top_pair[(w * k + i) * 2 + 1] = ok ? static_cast<int32_t>(c.i % R) : -1;
        }
        if (top_pair_value) top_pair_value[w * k + i] = ok ? c.v : 0;
      }
      prev = c.v > 0 ? c : VI{0, INT64_MAX};
    }
  }
  cluster.sync();  // the other CTAs' candidates stay in place until the merge has read them
}

// ---------------------------------------------------------------------------
// Gates (App. C).  One CTA per window: the CTA scans rank roles and splits the
// window's step leaders into 256 segments for the switch count; thread 0 then
// evaluates the gates with exact integer comparisons a*den <op> num*b.
constexpr int kGateThreads = 256;

__device__ __forceinline__ bool r_gt(__int128 lhs, sf_ratio r, __int128 rhs) {
  return lhs * r.den > static_cast<__int128>(r.num) * rhs;
}
__device__ __forceinline__ bool r_lt(__int128 lhs, sf_ratio r, __int128 rhs) {
  return lhs * r.den < static_cast<__int128>(r.num) * rhs;
}
__device__ __forceinline__ bool r_ge(__int128 lhs, sf_ratio r, __int128 rhs) {
  return lhs * r.den >= static_cast<__int128>(r.num) * rhs;
}

__global__ void __launch_bounds__(kGateThreads) gates_kernel(const GateJob g) {
  __shared__ int seg_e[kGateThreads], seg_sw[kGateThreads], seg_first[kGateThreads],
      seg_last[kGateThreads];
  const int64_t w = blockIdx.x;
  const int64_t S = g.S;
  const int64_t tb = w * g.W, te = min(tb + g.W, g.T), n = te - tb;
  int mixed = 0;
  if (g.role) {
    const int32_t r0 = g.role[0];
    for (int64_t r = 1 + threadIdx.x; r < g.R; r += kGateThreads) mixed |= g.role[r] != r0;
  }
  mixed = __syncthreads_or(mixed);
  {
    const int j = threadIdx.x;
    const int64_t sb = tb + n * j / kGateThreads, se = tb + n * (j + 1) / kGateThreads;
    int e = 0, sw = 0, first = -1, last = -1;
    for (int64_t t = sb; t < se; ++t) {
      const uint8_t sl = g.step_lead[t];
      if (sl & SF_STEP_CONFIDENT) {
        const int ld = sl & 31;
        if (last >= 0 && ld != last) ++sw;
        if (first < 0) first = ld;
        last = ld;
        ++e;
      }
    }
    seg_e[j] = e;
    seg_sw[j] = sw;
    seg_first[j] = first;
    seg_last[j] = last;
  }
  __syncthreads();
  if (threadIdx.x != 0) return;

  int64_t e = 0, sw = 0;
  int last = -1;
  for (int j = 0; j < kGateThreads; ++j) {
    if (seg_e[j] == 0) continue;
    e += seg_e[j];
    sw += seg_sw[j] + ((last >= 0 && seg_first[j] != last) ? 1 : 0);
    last = seg_last[j];
  }
  const sf_label_config& c = g.cfg;
  const bool high_switch = e >= 2 && r_ge(e, c.gamma_elig, n) && r_gt(sw, c.gamma_switch, e - 1);

  const int64_t* Xw = g.X + w * S;
  const int64_t* Yw = g.Y + w * S;
  const int64_t Dw = g.D[w];
  bool tel = g.missing != nullptr && g.missing[w] > c.max_missing_ranks;
  if (g.quality) {
    const uint64_t* q = g.quality + w * 6;
    const unsigned __int128 res = (static_cast<unsigned __int128>(q[1]) << 64) | q[0];
    const unsigned __int128 ovl = (static_cast<unsigned __int128>(q[3]) << 64) | q[2];
    const unsigned __int128 ws = (static_cast<unsigned __int128>(q[5]) << 64) | q[4];
    if (res * static_cast<uint64_t>(c.closure_max.den) > ws * static_cast<uint64_t>(c.closure_max.num)) tel = true;
    if (ovl * static_cast<uint64_t>(c.overlap_max.den) > ws * static_cast<uint64_t>(c.overlap_max.num)) tel = true;
  }
  const bool raw = Dw < c.denom_floor_ns || Dw == 0;
  if (raw) tel = true;
  uint32_t lab = SF_LABEL_FRONTIER_ACCOUNTING, route = 0, amb = 0;
  if (tel) lab |= SF_LABEL_TELEMETRY_LIMITED;
  if (mixed) lab |= SF_LABEL_ROLE_AWARE_NEEDED;
  if (raw) {
    lab |= SF_LABEL_RAW_ONLY;
  } else {
    int s1 = 0, g1 = 0;
    for (int s = 1; s < S; ++s) {
      if (Xw[s] > Xw[s1]) s1 = s;
      if (Yw[s] > Yw[g1]) g1 = s;
    }
    int nA = 0, nG = 0;
    for (int s = 0; s < S; ++s) {
      if (r_lt(Xw[s1] - Xw[s], c.eta_A, Dw)) {
        amb |= 1u << s;
        ++nA;
      }
      if (r_lt(Yw[g1] - Yw[s], c.eta_G, Dw)) {
        amb |= 1u << s;
        ++nG;
      }
    }
    __int128 cum = 0;
    for (int i = 0; i < S; ++i) {  // leading-share prefix reaching tau_C
      int pick = -1;
      for (int s = 0; s < S; ++s)
        if (!((route >> s) & 1u) && (pick < 0 || Xw[s] > Xw[pick])) pick = s;
      route |= 1u << pick;
      cum += Xw[pick];
      if (r_ge(cum, c.tau_C, Dw)) break;
    }
    const bool hiA = r_gt(Xw[s1], c.gamma_A, Dw);
    const bool loG = r_lt(Yw[s1], c.gamma_G, Dw);
    const bool W1 = (c.model_fit_mask >> s1) & 1u;
    const bool gain_tie = nG >= 2 && r_ge(Yw[g1], c.gamma_G, Dw);
    if (hiA && loG) lab |= W1 ? SF_LABEL_SYNC_WAIT_DEPENDENT : SF_LABEL_CO_CRITICAL;
    if (hiA && !loG) lab |= SF_LABEL_DIRECT_EXPOSURE;
    if (nA >= 2 || gain_tie || high_switch) {
      lab |= SF_LABEL_CO_CRITICAL;
      lab &= ~(SF_LABEL_DIRECT_EXPOSURE | SF_LABEL_SYNC_WAIT_DEPENDENT);
    }
    if (tel || mixed) lab &= ~(SF_LABEL_DIRECT_EXPOSURE | SF_LABEL_SYNC_WAIT_DEPENDENT);
  }
  g.labels[w] = lab;
  g.route_mask[w] = route;
  g.amb_mask[w] = amb;
  for (int s = 0; s < S; ++s) {
    if (g.share) g.share[w * S + s] = raw ? 0.0 : static_cast<double>(Xw[s]) / static_cast<double>(Dw);
    if (g.gain) g.gain[w * S + s] = raw ? 0.0 : static_cast<double>(Yw[s]) / static_cast<double>(Dw);
  }
  if (g.n_confident) g.n_confident[w] = static_cast<int32_t>(e);
  if (g.n_switch) g.n_switch[w] = static_cast<int32_t>(sw);
}

template <int NPL>
cudaError_t launch_median_npl(const int64_t* d, int64_t T, int64_t RS, int64_t W, int64_t nW,
                              int64_t ngroups, int64_t* m, cudaStream_t stream) {
  const size_t smem = size_t(kMedCols) * (32 * NPL + 1) * sizeof(int64_t) +
                      size_t(kMedCols) * kMedBins * sizeof(uint32_t);
  const bool vec = (RS % 2) == 0 && (reinterpret_cast<uintptr_t>(d) % 16) == 0;
  auto kern = vec ? median_kernel<NPL, true> : median_kernel<NPL, false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  kern<<<static_cast<unsigned>(nW * ngroups), kMedThreads, smem, stream>>>(d, T, RS, W, ngroups, m);
  return cudaGetLastError();
}

template <int NPL>
cudaError_t launch_median_tma(const CUtensorMap& map, int64_t T, int64_t RS, int64_t W, int64_t nW,
                              int64_t ngroups, int box_rows, int nbox, int64_t* m, uint32_t* status,
                              cudaStream_t stream) {
  const size_t tile_rows = std::max<size_t>(size_t(nbox) * box_rows, 32 * NPL);  // every slot's row is in the tile
  const size_t smem = 1024 + tile_rows * 64 + size_t(kMedCols) * kMedHistWords * 4 + 16;
  cudaError_t e =
      cudaFuncSetAttribute(median_tma_kernel<NPL>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  median_tma_kernel<NPL><<<static_cast<unsigned>(nW * ngroups), kMedThreads, smem, stream>>>(
      map, T, RS, W, ngroups, box_rows, nbox, static_cast<int>(tile_rows), m, status);
  return cudaGetLastError();
}

// Self-test of the bounded wait: every thread waits on an mbarrier phase
// that nothing completes (count 2, one arrival), so the wait must give up
// after limit_ns, record SF_ST_TIMEOUT and let the kernel finish.
__global__ void wait_selftest_kernel(uint64_t limit_ns, uint32_t* status) {
  __shared__ uint64_t bar;
  __shared__ int abort;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 2);
    abort = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_arrive(&bar);  // one of the two arrivals the phase needs
  const bool ok = mbar_wait_bounded(&bar, 0, &abort, limit_ns);
  if (threadIdx.x == 0) report(status, ok ? 0u : SF_ST_TIMEOUT);
}

}  // namespace

cudaError_t launch_wait_selftest(uint64_t limit_ns, uint32_t* status, cudaStream_t stream) {
  count_launch();
  wait_selftest_kernel<<<1, 64, 0, stream>>>(limit_ns, status);
  return cudaGetLastError();
}

cudaError_t launch_zero(void* p, size_t bytes, cudaStream_t stream) {
  if (bytes == 0) return cudaSuccess;
  const size_t words = bytes / 4;
  const int grid = static_cast<int>(std::min<size_t>((words + 255) / 256, size_t(sm_count()) * 8));
  count_launch();
  zero_kernel<<<grid, 256, 0, stream>>>(static_cast<uint32_t*>(p), words);
  return cudaGetLastError();
}

cudaError_t launch_window_median(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W,
                                 int64_t* m, uint32_t* status, cudaStream_t stream) {
  const int64_t RS = R * S;
  const int64_t nW = (T + W - 1) / W;
  const int64_t ngroups = (RS + kMedCols - 1) / kMedCols;
  const int64_t n = std::min(W, T);
  count_launch();
  // Bulk-copy path: rows of d are 16-byte multiples (RS even), d is 16-byte
  // aligned, windows fit the register path, the driver encoder is available.
  if (RS % 2 == 0 && reinterpret_cast<uintptr_t>(d) % 16 == 0 && n <= 1024 && T < (int64_t(1) << 31) &&
      encode_fn() != nullptr) {
    const int nbox = static_cast<int>((n + 255) / 256);
    const int box_rows = static_cast<int>(((n + nbox - 1) / nbox + 15) / 16 * 16);  // 1024-byte boxes
    CUtensorMap map;
    const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(RS), static_cast<cuuint64_t>(T)};
    const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(RS) * 8};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(kMedCols), static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t estride[2] = {1, 1};
    if (encode_fn()(&map, CU_TENSOR_MAP_DATA_TYPE_INT64, 2, const_cast<int64_t*>(d), gdim, gstride, box, estride,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS) {
      if (n <= 32) return launch_median_tma<1>(map, T, RS, W, nW, ngroups, box_rows, nbox, m, status, stream);
      if (n <= 64) return launch_median_tma<2>(map, T, RS, W, nW, ngroups, box_rows, nbox, m, status, stream);
      if (n <= 128) return launch_median_tma<4>(map, T, RS, W, nW, ngroups, box_rows, nbox, m, status, stream);
      if (n <= 256) return launch_median_tma<8>(map, T, RS, W, nW, ngroups, box_rows, nbox, m, status, stream);
      if (n <= 512) return launch_median_tma<16>(map, T, RS, W, nW, ngroups, box_rows, nbox, m, status, stream);
      return launch_median_tma<32>(map, T, RS, W, nW, ngroups, box_rows, nbox, m, status, stream);
    }
  }
  if (n <= 32) return launch_median_npl<1>(d, T, RS, W, nW, ngroups, m, stream);
  if (n <= 64) return launch_median_npl<2>(d, T, RS, W, nW, ngroups, m, stream);
  if (n <= 128) return launch_median_npl<4>(d, T, RS, W, nW, ngroups, m, stream);
  if (n <= 256) return launch_median_npl<8>(d, T, RS, W, nW, ngroups, m, stream);
  if (n <= 512) return launch_median_npl<16>(d, T, RS, W, nW, ngroups, m, stream);
  if (n <= 1024) return launch_median_npl<32>(d, T, RS, W, nW, ngroups, m, stream);
  median_global_kernel<<<static_cast<unsigned>(nW * ngroups), kMedThreads, 0, stream>>>(d, T, RS, W, ngroups, m);
  return cudaGetLastError();
}

cudaError_t launch_topk(const int64_t* X, const int64_t* E, int64_t nW, int64_t S, int64_t R, int32_t k,
                        int32_t* top_stage, int64_t* top_stage_value, int32_t* top_pair,
                        int64_t* top_pair_value, cudaStream_t stream) {
  count_launch();
  topk_kernel<<<static_cast<unsigned>(nW * kTopCluster), kTopThreads, 0, stream>>>(
      X, E, S, R, k, top_stage, top_stage_value, top_pair, top_pair_value);
  return cudaGetLastError();
}

cudaError_t launch_gates(const GateJob& job, cudaStream_t stream) {
  count_launch();
  gates_kernel<<<static_cast<unsigned>(job.nW), kGateThreads, 0, stream>>>(job);
  return cudaGetLastError();
}

}  // namespace sf

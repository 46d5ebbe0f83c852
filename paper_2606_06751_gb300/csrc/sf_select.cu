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

// Clears up to kZeroMax buffers in one launch (a call's accumulators), and
// lets the pass that follows it on the stream start at once (it waits for
// this kernel's completion before its first write).
__global__ void zero_many_kernel(const ZeroList z) {
  griddep_launch_dependents();
  for (int b = 0; b < z.n; ++b) {
    uint32_t* __restrict__ p = static_cast<uint32_t*>(z.ptr[b]);
    for (size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x; i < z.words[b];
         i += size_t(gridDim.x) * blockDim.x)
      p[i] = 0u;
  }
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
// Per-warp counters: 256 digit bins, then 48 spare words (a compacted bin of
// at most 32 values and its padding to whole 16-byte groups).  304 words =
// 1216 bytes keeps every warp's block 16-byte aligned.
constexpr int kMedHistWords = kMedBins + 48;

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

// Radix selection on a column held in registers (x[i] = row lane + 32 i):
// the k-th smallest of the live values, all below 2^nbits.  Padding slots
// must hold 2^nbits - 1: they sort at or after every live value, so counting
// them never moves the rank-k bin and no slot needs a validity test.  The
// first digit is the top 8 bits of the range, [nbits - 8, nbits), so it
// spreads over the 256 bins and its chosen bin usually holds a few percent of
// the column; each later pass counts, predicated, the values that share the
// digits chosen so far.  As soon as the chosen bin holds at most 32 values
// they are compacted into the spare words after the bins (ballot ranks, no
// atomics) and each is ranked by counting.
template <int NPL>
__device__ __forceinline__ uint32_t warp_select_regs(const uint32_t (&x)[NPL], int nbits, uint32_t k,
                                                     uint32_t* hist, int lane) {
  uint32_t prefix = 0, rem = k;
  int hi = nbits;
  bool first = true;
  while (hi > 0) {
    const int sh = hi > 8 ? hi - 8 : 0;
    const uint32_t mask = (1u << (hi - sh)) - 1u;
    reinterpret_cast<uint4*>(hist)[2 * lane] = make_uint4(0, 0, 0, 0);
    reinterpret_cast<uint4*>(hist)[2 * lane + 1] = make_uint4(0, 0, 0, 0);
    __syncwarp();
    if (first) {
#pragma unroll
      for (int i = 0; i < NPL; ++i) atomicAdd(&hist[x[i] >> sh], 1u);  // x < 2^nbits: the bin is below 256
    } else {
#pragma unroll
      for (int i = 0; i < NPL; ++i)
        red_shared_inc_if(&hist[(x[i] >> sh) & mask], (x[i] >> hi) == (prefix >> hi));
    }
    __syncwarp();
    uint32_t digit, below;
    hist_find(hist, rem, lane, digit, below);
    const uint32_t kept = hist[digit];
    rem -= below;
    prefix |= digit << sh;
    hi = sh;
    first = false;
    if (hi > 0 && kept <= 32) {
      uint32_t* cbuf = hist + kMedBins;
      const uint32_t below_lane = (1u << lane) - 1u;
      uint32_t base = 0;
#pragma unroll
      for (int i = 0; i < NPL; ++i) {
        const bool mt = (x[i] >> hi) == (prefix >> hi);
        const uint32_t mm = __ballot_sync(kFull, mt);
        if (mm) {
          if (mt) cbuf[base + __popc(mm & below_lane)] = x[i];
          base += __popc(mm);
        }
      }
      if (lane < 3) cbuf[kept + lane] = 0xffffffffu;  // pad to whole 16-byte groups (kept + 3 <= 35 < 64 spare)
      __syncwarp();
      // rank each bin value by counting (broadcast reads of the bin): the
      // answer is a value with lt <= rem < le.  Padding counts only toward
      // le of the largest key, which no rank below kept can need.
      const uint32_t v = cbuf[lane & 31];
      uint32_t lt = 0, le = 0;
      for (uint32_t q = 0; q < kept; q += 4) {
        const uint4 c = *reinterpret_cast<const uint4*>(cbuf + q);
        lt += (c.x < v) + (c.y < v) + (c.z < v) + (c.w < v);
        le += (c.x <= v) + (c.y <= v) + (c.z <= v) + (c.w <= v);
      }
      const uint32_t hit = __ballot_sync(kFull, static_cast<uint32_t>(lane) < kept && lt <= rem && rem < le);
      const uint32_t ans = __shfl_sync(kFull, v, __ffs(hit) - 1);
      __syncwarp();
      return ans;
    }
    __syncwarp();
  }
  return prefix;
}

// Lower median of one column of n <= 32 NPL rows read from global memory
// (stride RS) on every pass, on 64-bit order-preserving keys: the path of a
// column whose values do not share their high 32 bits.  Kept out of line so
// its registers do not weigh on the 32-bit path.
template <int NPL>
__device__ __noinline__ int64_t median_column_global(const int64_t* __restrict__ dc, int64_t RS, int n, uint32_t* hist,
                                                     int lane) {
  constexpr uint64_t kSign = 1ull << 63;
  auto ukey = [&](int i) { return static_cast<uint64_t>(__ldg(dc + int64_t(lane + 32 * i) * RS)) ^ kSign; };
  uint64_t lo = ~0ull, hi = 0;
#pragma unroll 4
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
  const uint32_t k = static_cast<uint32_t>((n - 1) / 2);
  const uint64_t key =
      lo + warp_radix_select<uint64_t, NPL>([&](int i) { return ukey(i) - lo; }, n, nbits, k, hist, lane);
  return static_cast<int64_t>(key ^ kSign);
}

// Persistent form of the median: each CTA walks (window, 8-column) tiles
// with one tile buffer and two mbarriers.  `full` completes when a tile's
// bulk copies have landed; each warp copies its column into registers and
// arrives on `empty`, and once all eight have, one thread issues the copies
// of the CTA's next tile into the same buffer, so the copy runs under the
// selection of the current tile and no CTA-wide barrier aligns the warps.
// The selection touches only registers and the warp's counters.  A column
// whose values do not share their high 32 bits selects on 64-bit values
// re-read from d.  Every window of a launch holds the same n rows.
template <int NPL, bool kFit>
__global__ void __launch_bounds__(kMedThreads, 3)
    median_persist_kernel(const __grid_constant__ CUtensorMap map, const int64_t* __restrict__ d, int64_t T,
                          int64_t RS, int64_t W, int64_t w0, int64_t nW, int64_t ngroups, int box_rows, int nbox,
                          int64_t* __restrict__ m, uint32_t* status) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* tile = align_1024(smem_raw);
  const uint32_t tile_bytes = uint32_t(nbox) * uint32_t(box_rows) * 64u;  // bytes the copies write
  const int tile_rows = max(nbox * box_rows, 32 * NPL);
  uint32_t* hists = reinterpret_cast<uint32_t*>(tile + uint32_t(tile_rows) * 64u);
  uint64_t* full = reinterpret_cast<uint64_t*>(hists + kMedCols * kMedHistWords);
  uint64_t* empty = full + 1;
  volatile int* abort = reinterpret_cast<volatile int*>(full + 2);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint32_t* hist = hists + warp * kMedHistWords;
  const int64_t ntiles = nW * ngroups;
  auto issue = [&](int64_t id) {  // one thread: the bulk copies of tile `id`
    const int64_t c0 = (id % ngroups) * kMedCols;
    const int64_t tb = (w0 + id / ngroups) * W;
    mbar_arrive_expect_tx(full, tile_bytes);
    for (int b = 0; b < nbox; ++b)
      tma_load_2d(tile + size_t(b) * box_rows * 64, &map, static_cast<int32_t>(c0),
                  static_cast<int32_t>(tb + int64_t(b) * box_rows), full);
  };
  if (threadIdx.x == 0) {
    mbar_init(full, 1);
    mbar_init(empty, kMedCols);
    *abort = 0;
    fence_barrier_init();
  }
  __syncthreads();
  bool issued = blockIdx.x < ntiles;  // (thread 0) the copies of the awaited tile were issued
  if (threadIdx.x == 0 && issued) issue(blockIdx.x);
  const unsigned char* col = tile + lane * 64u + ((((warp >> 1) ^ ((lane >> 1) & 3)) << 4) | ((warp & 1) << 3));
  uint32_t phase = 0;
  for (int64_t id = blockIdx.x; id < ntiles; id += gridDim.x, phase ^= 1u) {
    const int64_t w = w0 + id / ngroups;
    const int64_t c0 = (id % ngroups) * kMedCols;
    const bool mine = warp < imin64(kMedCols, RS - c0);
    const int n = static_cast<int>(imin64(W, T - w * W));
    // a warp goes on only if all its lanes saw the tile (a wait gives up
    // after its time limit, or at once when another thread has)
    if (!__all_sync(kFull, mbar_wait_bounded(full, phase, abort))) {
      if (threadIdx.x == 0) {
        report(status, SF_ST_TIMEOUT);
        if (issued) mbar_wait_timeout(full, phase);  // let the copies land before the CTA's memory is released
      }
      return;
    }
    // Slot i holds a row of the window iff lane + 32 i < n (with kFit, only
    // the last slot can fail it).  A padding slot repeats a live value; the
    // high words agree iff their AND equals their OR over the column.
    auto live = [&](int i) { return (kFit && i + 1 < NPL) || lane + 32 * i < n; };
    uint32_t xl[NPL];
    uint32_t hand = 0xffffffffu, hor = 0u, live_x = 0u;
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
      const uint2 v = *reinterpret_cast<const uint2*>(col + i * 2048);  // in the tile even past the window
      if (i == 0) live_x = kFit && NPL >= 2 ? v.x : __shfl_sync(kFull, v.x, 0);  // row 0 is in every window
      const bool okr = live(i);
      xl[i] = okr ? v.x : live_x;
      hand &= okr ? v.y : 0xffffffffu;
      hor |= okr ? v.y : 0u;
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(empty);  // this warp is done with the buffer
    const int64_t next = id + gridDim.x;
    if (threadIdx.x == 0 && next < ntiles) {
      issued = mbar_wait_bounded(empty, phase, abort);
      if (issued) issue(next);  // else the abort flag is set and every warp leaves at its next wait
    }
    if (!mine) continue;
    const uint32_t hw = __reduce_and_sync(kFull, hand);
    const uint32_t k = static_cast<uint32_t>((n - 1) / 2);
    if (hw == __reduce_or_sync(kFull, hor)) {
      uint32_t lmin = xl[0], lmax = xl[0];
#pragma unroll
      for (int i = 1; i + 1 < NPL; i += 2) {
        lmin = __vimin3_u32(lmin, xl[i], xl[i + 1]);
        lmax = __vimax3_u32(lmax, xl[i], xl[i + 1]);
      }
      if ((NPL & 1) == 0) {
        lmin = min(lmin, xl[NPL - 1]);
        lmax = max(lmax, xl[NPL - 1]);
      }
      lmin = __reduce_min_sync(kFull, lmin);
      lmax = __reduce_max_sync(kFull, lmax);
      const uint32_t range = lmax - lmin;
      const int nbits = range ? 32 - __clz(static_cast<int>(range)) : 0;
      const uint32_t pad = nbits == 32 ? 0xffffffffu : (1u << nbits) - 1u;  // sorts at or after every live value
#pragma unroll
      for (int i = 0; i < NPL; ++i) xl[i] = live(i) ? xl[i] - lmin : pad;
      const uint32_t ans = warp_select_regs<NPL>(xl, nbits, k, hist, lane);
      if (lane == 0) m[w * RS + c0 + warp] = static_cast<int64_t>((static_cast<uint64_t>(hw) << 32) | (lmin + ans));
    } else {
      // the buffer may already hold the next tile: re-read the column from d
      const int64_t med = median_column_global<NPL>(d + w * W * RS + c0 + warp, RS, n, hist, lane);
      if (lane == 0) m[w * RS + c0 + warp] = med;
    }
  }
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
cudaError_t launch_median_tma(const CUtensorMap& map, const int64_t* d, int64_t T, int64_t RS, int64_t W,
                              int64_t w0, int64_t nW, int64_t n, int64_t ngroups, int box_rows, int nbox, int64_t* m, uint32_t* status,
                              cudaStream_t stream) {
  const size_t tile_rows = std::max<size_t>(size_t(nbox) * box_rows, 32 * NPL);  // every slot's row is in the tile
  const size_t smem = 1024 + tile_rows * 64 + size_t(kMedCols) * kMedHistWords * 4 + 32;  // + 2 mbarriers, flag
  auto kern = n > 32 * (NPL - 1) ? median_persist_kernel<NPL, true> : median_persist_kernel<NPL, false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kMedThreads, smem);
  if (e != cudaSuccess) return e;
  const int64_t grid = std::min<int64_t>(nW * ngroups, int64_t(sm_count()) * std::max(per_sm, 1));
  count_launch();
  kern<<<static_cast<unsigned>(grid), kMedThreads, smem, stream>>>(map, d, T, RS, W, w0, nW, ngroups, box_rows,
                                                                   nbox, m, status);
  return cudaGetLastError();
}

// Windows [w0, w0 + nW) that each hold n rows: the tensor map's box covers a
// window in up to four 256-row copies; NPL slots per lane hold n rows.
cudaError_t launch_median_windows(const int64_t* d, int64_t T, int64_t RS, int64_t W, int64_t w0, int64_t nW,
                                  int64_t n, int64_t ngroups, int64_t* m, uint32_t* status, cudaStream_t stream,
                                  bool& done) {
  done = false;
  const int nbox = static_cast<int>((n + 255) / 256);
  const int box_rows = static_cast<int>(((n + nbox - 1) / nbox + 15) / 16 * 16);  // 1024-byte boxes
  CUtensorMap map;
  const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(RS), static_cast<cuuint64_t>(T)};
  const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(RS) * 8};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kMedCols), static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estride[2] = {1, 1};
  if (encode_fn()(&map, CU_TENSOR_MAP_DATA_TYPE_INT64, 2, const_cast<int64_t*>(d), gdim, gstride, box, estride,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaSuccess;
  done = true;
  if (n <= 32) return launch_median_tma<1>(map, d, T, RS, W, w0, nW, n, ngroups, box_rows, nbox, m, status, stream);
  if (n <= 64) return launch_median_tma<2>(map, d, T, RS, W, w0, nW, n, ngroups, box_rows, nbox, m, status, stream);
  if (n <= 128) return launch_median_tma<4>(map, d, T, RS, W, w0, nW, n, ngroups, box_rows, nbox, m, status, stream);
  if (n <= 256) return launch_median_tma<8>(map, d, T, RS, W, w0, nW, n, ngroups, box_rows, nbox, m, status, stream);
  if (n <= 512) return launch_median_tma<16>(map, d, T, RS, W, w0, nW, n, ngroups, box_rows, nbox, m, status, stream);
  return launch_median_tma<32>(map, d, T, RS, W, w0, nW, n, ngroups, box_rows, nbox, m, status, stream);
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

cudaError_t launch_zero_many(const ZeroList& z, cudaStream_t stream, bool* launched) {
  size_t words = 0;
  for (int b = 0; b < z.n; ++b) words = std::max(words, z.words[b]);
  if (launched) *launched = false;
  if (words == 0) return cudaSuccess;
  if (launched) *launched = true;
  const int grid = static_cast<int>(std::min<size_t>((words + 255) / 256, size_t(sm_count()) * 8));
  count_launch();
  zero_many_kernel<<<grid, 256, 0, stream>>>(z);
  return cudaGetLastError();
}

cudaError_t launch_window_median(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W,
                                 int64_t* m, uint32_t* status, cudaStream_t stream) {
  const int64_t RS = R * S;
  const int64_t nW = (T + W - 1) / W;
  const int64_t ngroups = (RS + kMedCols - 1) / kMedCols;
  const int64_t n = std::min(W, T);
  // Bulk-copy path: rows of d are 16-byte multiples (RS even), d is 16-byte
  // aligned, windows fit the register path, the driver encoder is available.
  // A launch's windows share one row count (the slot tests depend on it), so
  // a short last window gets its own launch.
  if (RS % 2 == 0 && reinterpret_cast<uintptr_t>(d) % 16 == 0 && n <= 1024 && T < (int64_t(1) << 31) &&
      encode_fn() != nullptr) {
    const int64_t n_last = T - (nW - 1) * W;
    const int64_t nW_first = n_last == n ? nW : nW - 1;
    bool done = false;
    cudaError_t e = launch_median_windows(d, T, RS, W, 0, nW_first, n, ngroups, m, status, stream, done);
    if (e != cudaSuccess) return e;
    if (done && nW_first == nW) return cudaSuccess;
    if (done) {
      e = launch_median_windows(d, T, RS, W, nW - 1, 1, n_last, ngroups, m, status, stream, done);
      if (e != cudaSuccess || done) return e;
    }
    // no tensor map: every window goes the plain-load way below
  }
  count_launch();
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

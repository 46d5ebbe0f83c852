// sf_rank.cu - cross-rank order statistics per (step, stage): the lower
// median over ranks of the prefixes P[t,r,s] (for the lag of Sec. 4) or of the
// durations d[t,r,s] (for the raw rank spread of the Sec. 6 routing table),
// with the maximum and the second largest value.
//
// The steps are processed in chunks whose scratch stays in L2; per chunk two
// kernels run, the encode of the next chunk overlapping the select of this
// one (programmatic dependent launch, two scratch buffers):
//  encode (rank_encode_split_kernel for 4, 8 or 16 stages, a rank row split
//    over S/2 lanes; rank_encode_kernel, a row per thread, otherwise) -
//    streams the chunk's rank rows once from HBM with streaming loads, so
//    that d does not push the scratch out of L2, and writes every (step,
//    stage) column as 32-bit keys: the value minus rank 0's value, sign bit
//    flipped, so that unsigned key order is value order.  A persistent grid
//    walks blocks of 1024 rank rows of one step and writes each block's
//    minimum, maximum and second largest key per stage and a flag for a value
//    2^31 or more away from rank 0's (that step then takes the 64-bit path).
//    A warp whose values are all small works in 32-bit arithmetic.
//  rank_select_kernel - one CTA per (step, stage) column at a time: radix
//    selection on the key offsets from the column minimum.  The first pass
//    reads the column from L2 four keys at a time into a 2048-bin histogram
//    of the top 11 bits of the range.  A chosen bin of at most 32 keys is
//    gathered by a second read and ranked by counting in one warp; a fuller
//    bin is kept as candidates by the second read, so later 8-bit passes read
//    only those.  Once a column has been read for the last time its L2 lines
//    are discarded, so the dead scratch is never written back to HBM.
// A last small kernel forms delta-lag from the lag.
#include <algorithm>
#include <cstdint>

#include "sf_device.cuh"
#include "sf_launch.h"

namespace sf {
namespace {

constexpr int kRkMaxS = 32;
constexpr int kEncThreads = 256;
constexpr int kEncRows = 1024;  // rank rows per encode item (4 per thread)
constexpr int kSelThreads = 128;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kSelPerSM = 1536 / kSelThreads;  // resident select CTAs per SM
constexpr int kSelCand = 2048;  // candidate keys a column may keep after the second pass
constexpr size_t kRkChunkTarget = size_t(52) << 20;  // scratch of one chunk buffer; two fit L2 (52 MB: 207 steps of 8192 x 8, one select wave)

struct RankParams {
  const int64_t* d;
  int64_t T, R, S;
  int of_prefix;  // 1: order statistics of P (lag); 0: of d (spread)
  int64_t t0, W, w_first;
  int64_t *L, *G;    // [T][S], nullable
  int64_t *Lw, *Gw;  // [nW][S] window sums of L and G, nullable
  int64_t* spread;   // [nW][S], nullable
  uint32_t* status;
  // one chunk of steps [c0, c0 + Tc) and its scratch
  int64_t c0, Tc;
  int64_t ldR;     // key column stride: R rounded up to 32 (whole 128-byte lines)
  int nblk;        // encode blocks per step
  uint32_t* keys;  // [Tc][S][ldR]
  uint32_t* pmin;  // [Tc][nblk][S]
  uint32_t* pmax;  // [Tc][nblk][S]
  uint32_t* psec;  // [Tc][nblk][S] second largest key of the block (a tie counts)
  uint32_t* pbad;  // [Tc][nblk]
  int64_t* ref;    // [Tc][S] rank 0's value
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

__device__ __forceinline__ int64_t key_value(int64_t ref, uint32_t key) {
  return ref + static_cast<int64_t>(static_cast<int32_t>(key ^ 0x80000000u));
}

// Programmatic dependent launch: the encode of chunk c+1 runs while the
// select of chunk c does; each kernel waits for its predecessor in the stream
// only where it must (see launch_rank_select).

__device__ __forceinline__ void discard_l2_line(const void* p) {
  asm volatile("discard.global.L2 [%0], 128;" ::"l"(p) : "memory");
}

// ------------------------------------------------------------------ encode

template <int SC>
__global__ void __launch_bounds__(kEncThreads) rank_encode_kernel(const RankParams p) {
  constexpr int kCols = SC > 0 ? SC : kRkMaxS;
  constexpr int kWarps = kEncThreads / 32;
  __shared__ int64_t sref[kRkMaxS];
  __shared__ uint32_t wmn[kWarps][kRkMaxS], wmx[kWarps][kRkMaxS], wm2[kWarps][kRkMaxS];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int S = SC > 0 ? SC : static_cast<int>(p.S);
  const int64_t R = p.R;
  uint32_t dor = 0, tor = 0;
  const int64_t items = p.Tc * p.nblk;
  for (int64_t item = blockIdx.x; item < items; item += gridDim.x) {
    const int64_t tl = item / p.nblk;
    const int blk = static_cast<int>(item - tl * p.nblk);
    const int64_t* dt = p.d + (p.c0 + tl) * R * S;
    if (warp == 0) {
      // rank 0's values: the reference of the step's keys
      int64_t x = lane < S ? __ldg(dt + lane) : 0;
      if (p.of_prefix) {
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int64_t up = __shfl_up_sync(kFull, x, o);
          if (lane >= o) x += up;
        }
      }
      if (lane < S) {
        sref[lane] = x;
        if (blk == 0) p.ref[tl * S + lane] = x;
      }
    }
    __syncthreads();
    uint32_t mn[kCols], m1[kCols], m2[kCols];
#pragma unroll
    for (int s = 0; s < kCols; ++s) {
      mn[s] = 0xffffffffu;
      m1[s] = 0u;
      m2[s] = 0u;
    }
    bool bad = false;
    const int64_t rb = int64_t(blk) * kEncRows;
    const int nrows = static_cast<int>(R - rb < kEncRows ? R - rb : kEncRows);
    uint32_t* kt = p.keys + tl * S * p.ldR + rb;
    // one row of this thread: stage values -> keys and column statistics
    auto encode_row = [&](const int64_t* v, int i) {
      int64_t P = 0;
#pragma unroll
      for (int s = 0; s < kCols; ++s) {
        if (s >= S) break;
        dor |= static_cast<uint32_t>(static_cast<uint64_t>(v[s]) >> 32);
        P += v[s];
        const int64_t diff = (p.of_prefix ? P : v[s]) - sref[s];
        bad |= (static_cast<uint64_t>(diff + 0x80000000ll) >> 32) != 0;
        const uint32_t k = static_cast<uint32_t>(diff) ^ 0x80000000u;
        kt[s * p.ldR + i] = k;
        mn[s] = k < mn[s] ? k : mn[s];
        top2_merge<uint32_t>(m1[s], m2[s], k, 0u);
      }
      tor |= static_cast<uint32_t>(static_cast<uint64_t>(P) >> 32);
    };
    if constexpr (SC > 0 && SC % 2 == 0 && SC <= 10) {
      // two rows' loads in flight per thread
      for (int i = tid; i < nrows; i += 2 * kEncThreads) {
        const bool two = i + kEncThreads < nrows;
        int64_t a[SC], b[SC];
        const longlong2* ra = reinterpret_cast<const longlong2*>(dt + (rb + i) * S);
        const longlong2* rbp = reinterpret_cast<const longlong2*>(dt + (rb + i + (two ? kEncThreads : 0)) * S);
#pragma unroll
        for (int h = 0; h < SC / 2; ++h) {
          const longlong2 x = __ldcs(ra + h);
          const longlong2 y = __ldcs(rbp + h);
          a[2 * h] = x.x;
          a[2 * h + 1] = x.y;
          b[2 * h] = y.x;
          b[2 * h + 1] = y.y;
        }
        encode_row(a, i);
        if (two) encode_row(b, i + kEncThreads);
      }
    } else {
      for (int i = tid; i < nrows; i += kEncThreads) {
        const int64_t* row = dt + (rb + i) * S;
        int64_t v[kCols];
#pragma unroll
        for (int s = 0; s < kCols; ++s) {
          if (s >= S) break;
          v[s] = __ldcs(row + s);
        }
        encode_row(v, i);
      }
    }
    // block minimum, maximum and second largest per column: warp, then CTA
#pragma unroll
    for (int s = 0; s < kCols; ++s) {
      if (SC == 0 && s >= S) break;
      uint32_t a1 = m1[s], a2 = m2[s];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const uint32_t o1 = __shfl_xor_sync(kFull, a1, o);
        const uint32_t o2 = __shfl_xor_sync(kFull, a2, o);
        top2_merge<uint32_t>(a1, a2, o1, o2);
      }
      const uint32_t a = __reduce_min_sync(kFull, mn[s]);
      if (lane == 0) {
        wmn[warp][s] = a;
        wmx[warp][s] = a1;
        wm2[warp][s] = a2;
      }
    }
    const int any_bad = __syncthreads_or(bad ? 1 : 0);
    if (tid < S) {
      uint32_t a = wmn[0][tid], a1 = wmx[0][tid], a2 = wm2[0][tid];
      for (int w = 1; w < kWarps; ++w) {
        a = wmn[w][tid] < a ? wmn[w][tid] : a;
        top2_merge<uint32_t>(a1, a2, wmx[w][tid], wm2[w][tid]);
      }
      p.pmin[item * S + tid] = a;
      p.pmax[item * S + tid] = a1;
      p.psec[item * S + tid] = a2;
    }
    if (tid == 0) p.pbad[item] = static_cast<uint32_t>(any_bad);
    __syncthreads();  // sref and the warp partials are rewritten by the next item
  }
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), p.of_prefix ? __reduce_or_sync(kFull, tor) : 0u);
  if (lane == 0) report(p.status, bits);
  // let this chunk's select launch, then finish only once the previous
  // chunk's select (which read the other scratch buffer) has finished, so
  // that this kernel's completion implies every earlier kernel's
  griddep_launch_dependents();
  griddep_wait();
}

// Encode with a rank row split over SC/2 lanes (SC = 4, 8 or 16): lane j of a
// group holds stages 2j and 2j+1 (one 16-byte load), the stage prefix comes
// from a segmented warp scan of the pair sums, and each thread keeps the
// statistics of its two columns only.  Few registers per thread let many
// CTAs, and four loads per thread, be in flight on each SM.
template <int SC>
__global__ void __launch_bounds__(kEncThreads) rank_encode_split_kernel(const RankParams p) {
  constexpr int L = SC / 2;                     // lanes per rank row
  constexpr int kRowsPerPass = kEncThreads / L;  // rows the CTA covers per pass
  constexpr int kUnroll = 4;                     // passes whose loads are in flight together
  constexpr int kWarps = kEncThreads / 32;
  // values below 2^kNarrowBits: a row's prefixes stay below SC * 2^kNarrowBits <= 2^31
  constexpr int kNarrowBits = SC <= 4 ? 29 : SC <= 8 ? 28 : 27;
  __shared__ int64_t sref[kRkMaxS];
  __shared__ uint32_t wmn[kWarps][kRkMaxS], wmx[kWarps][kRkMaxS], wm2[kWarps][kRkMaxS];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int j = lane % L;                      // this thread's stage pair
  const int rsub = tid / L;                    // this thread's row within a pass
  const int64_t R = p.R;
  uint32_t dor = 0, tor = 0;
  const int64_t items = p.Tc * p.nblk;
  for (int64_t item = blockIdx.x; item < items; item += gridDim.x) {
    const int64_t tl = item / p.nblk;
    const int blk = static_cast<int>(item - tl * p.nblk);
    const int64_t* dt = p.d + (p.c0 + tl) * R * SC;
    if (warp == 0) {
      int64_t x = lane < SC ? __ldg(dt + lane) : 0;
      if (p.of_prefix) {
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int64_t up = __shfl_up_sync(kFull, x, o);
          if (lane >= o) x += up;
        }
      }
      if (lane < SC) {
        sref[lane] = x;
        if (blk == 0) p.ref[tl * SC + lane] = x;
      }
    }
    __syncthreads();
    const int64_t ref0 = sref[2 * j], ref1 = sref[2 * j + 1];
    bool ref_narrow = true;  // rank 0's values (or prefixes) all in [0, 2^31)
#pragma unroll
    for (int q = 0; q < SC; ++q) ref_narrow &= (static_cast<uint64_t>(sref[q]) >> 31) == 0;
    uint32_t mn0 = 0xffffffffu, a0 = 0u, b0 = 0u, mn1 = 0xffffffffu, a1 = 0u, b1 = 0u;
    bool bad = false;
    const int64_t rb = int64_t(blk) * kEncRows;
    const int nrows = static_cast<int>(R - rb < kEncRows ? R - rb : kEncRows);
    uint32_t* k0 = p.keys + (tl * SC + 2 * j) * p.ldR + rb;
    uint32_t* k1 = k0 + p.ldR;
    const longlong2* base = reinterpret_cast<const longlong2*>(dt + rb * SC) + j;
    for (int r0 = 0; r0 < nrows; r0 += kUnroll * kRowsPerPass) {
      longlong2 v[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int r = r0 + u * kRowsPerPass + rsub;
        v[u] = r < nrows ? __ldcs(base + int64_t(r) * L) : make_longlong2(0, 0);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int r = r0 + u * kRowsPerPass + rsub;
        const bool live = r < nrows;
        const uint32_t hw = static_cast<uint32_t>(static_cast<uint64_t>(v[u].x) >> 32) |
                            static_cast<uint32_t>(static_cast<uint64_t>(v[u].y) >> 32);
        // 32-bit arithmetic when every value of the warp's rows is below
        // 2^kNarrowBits and so is rank 0's row: prefixes then stay below 2^31
        // and every key difference is exact in 32 bits
        const bool narrow = __all_sync(kFull, ((hw | ((static_cast<uint32_t>(v[u].x) |
                                                     static_cast<uint32_t>(v[u].y)) >> kNarrowBits)) == 0) &&
                                                  ref_narrow);
        if (narrow) {
          uint32_t y0 = static_cast<uint32_t>(v[u].x), y1 = static_cast<uint32_t>(v[u].y);
          if (p.of_prefix) {
            const uint32_t pair = y0 + y1;
            uint32_t incl = pair;
#pragma unroll
            for (int o = 1; o < L; o <<= 1) {
              const uint32_t up = __shfl_up_sync(kFull, incl, o, L);
              if (j >= o) incl += up;
            }
            y0 += incl - pair;
            y1 = incl;
          }
          const uint32_t q0 = (y0 - static_cast<uint32_t>(ref0)) ^ 0x80000000u;
          const uint32_t q1 = (y1 - static_cast<uint32_t>(ref1)) ^ 0x80000000u;
          if (live) {
            k0[r] = q0;
            k1[r] = q1;
            mn0 = q0 < mn0 ? q0 : mn0;
            mn1 = q1 < mn1 ? q1 : mn1;
            top2_merge<uint32_t>(a0, b0, q0, 0u);
            top2_merge<uint32_t>(a1, b1, q1, 0u);
          }
          continue;
        }
        dor |= hw;
        int64_t x0 = v[u].x, x1 = v[u].y;
        if (p.of_prefix) {
          // prefix before this pair: scan of the pair sums over the row's lanes
          const int64_t pair = x0 + x1;
          int64_t incl = pair;
#pragma unroll
          for (int o = 1; o < L; o <<= 1) {
            const int64_t up = __shfl_up_sync(kFull, incl, o, L);
            if (j >= o) incl += up;
          }
          x0 += incl - pair;
          x1 = incl;
          if (j == L - 1) tor |= static_cast<uint32_t>(static_cast<uint64_t>(incl) >> 32);
        }
        const int64_t d0 = x0 - ref0, d1 = x1 - ref1;
        const uint32_t q0 = static_cast<uint32_t>(d0) ^ 0x80000000u, q1 = static_cast<uint32_t>(d1) ^ 0x80000000u;
        if (live) {
          bad |= ((static_cast<uint64_t>(d0 + 0x80000000ll) | static_cast<uint64_t>(d1 + 0x80000000ll)) >> 32) != 0;
          k0[r] = q0;
          k1[r] = q1;
          mn0 = q0 < mn0 ? q0 : mn0;
          mn1 = q1 < mn1 ? q1 : mn1;
          top2_merge<uint32_t>(a0, b0, q0, 0u);
          top2_merge<uint32_t>(a1, b1, q1, 0u);
        }
      }
    }
    // merge the lanes of equal j (offsets that are multiples of L), then the warps
#pragma unroll
    for (int o = L; o < 32; o <<= 1) {
      mn0 = min(mn0, __shfl_xor_sync(kFull, mn0, o));
      mn1 = min(mn1, __shfl_xor_sync(kFull, mn1, o));
      const uint32_t oa0 = __shfl_xor_sync(kFull, a0, o), ob0 = __shfl_xor_sync(kFull, b0, o);
      const uint32_t oa1 = __shfl_xor_sync(kFull, a1, o), ob1 = __shfl_xor_sync(kFull, b1, o);
      top2_merge<uint32_t>(a0, b0, oa0, ob0);
      top2_merge<uint32_t>(a1, b1, oa1, ob1);
    }
    if (lane < L) {
      wmn[warp][2 * j] = mn0;
      wmx[warp][2 * j] = a0;
      wm2[warp][2 * j] = b0;
      wmn[warp][2 * j + 1] = mn1;
      wmx[warp][2 * j + 1] = a1;
      wm2[warp][2 * j + 1] = b1;
    }
    const int any_bad = __syncthreads_or(bad ? 1 : 0);
    if (tid < SC) {
      uint32_t a = wmn[0][tid], x1 = wmx[0][tid], x2 = wm2[0][tid];
      for (int w = 1; w < kWarps; ++w) {
        a = wmn[w][tid] < a ? wmn[w][tid] : a;
        top2_merge<uint32_t>(x1, x2, wmx[w][tid], wm2[w][tid]);
      }
      p.pmin[item * SC + tid] = a;
      p.pmax[item * SC + tid] = x1;
      p.psec[item * SC + tid] = x2;
    }
    if (tid == 0) p.pbad[item] = static_cast<uint32_t>(any_bad);
    __syncthreads();  // sref and the warp partials are rewritten by the next item
  }
  const uint32_t bits = range_bits(__reduce_or_sync(kFull, dor), p.of_prefix ? __reduce_or_sync(kFull, tor) : 0u);
  if (lane == 0) report(p.status, bits);
  griddep_launch_dependents();
  griddep_wait();
}

// ------------------------------------------------------------------ select

struct SelShared {
  uint32_t hist[256];
  uint32_t cand[kSelCand];
  int64_t wmin[kSelWarps], wmax[kSelWarps], wsec[kSelWarps];  // 64-bit path
  int64_t lo64;
  uint64_t pref64;
  uint32_t lo, hi, pref, rem, ncand, bad, sec_key, kept;
  int nb, compact, bytes64;
  int64_t med, F, sec;
};

// The 64-bit path for one column of a step whose values lie 2^31 or more
// from rank 0's: the values are re-read (and the prefix re-summed) from d in
// each pass; one pass per byte of the range.  Leaves med, F, sec in sh.
__device__ __noinline__ void select_column_64(const RankParams& p, int64_t t, int s, SelShared& sh) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int S = static_cast<int>(p.S);
  const int64_t R = p.R;
  const int64_t* dt = p.d + t * R * S;
  auto value = [&](int64_t r) {
    const int64_t* row = dt + r * S;
    if (!p.of_prefix) return __ldg(row + s);
    int64_t P = 0;
    for (int i = 0; i <= s; ++i) P += __ldg(row + i);
    return P;
  };
  int64_t a = INT64_MAX, x1 = -1, x2 = -1;
  for (int64_t r = tid; r < R; r += kSelThreads) {
    const int64_t x = value(r);
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
    sh.wmin[warp] = a;
    sh.wmax[warp] = x1;
    sh.wsec[warp] = x2;
  }
  __syncthreads();
  if (tid == 0) {
    a = sh.wmin[0];
    x1 = sh.wmax[0];
    x2 = sh.wsec[0];
    for (int w = 1; w < kSelWarps; ++w) {
      a = sh.wmin[w] < a ? sh.wmin[w] : a;
      top2_merge<int64_t>(x1, x2, sh.wmax[w], sh.wsec[w]);
    }
    sh.lo64 = a;
    sh.F = x1;
    sh.sec = R >= 2 ? x2 : x1;
    const uint64_t range = static_cast<uint64_t>(x1 - a);
    sh.bytes64 = range ? (64 - __clzll(static_cast<long long>(range)) + 7) / 8 : 0;
    sh.pref64 = 0;
    sh.rem = static_cast<uint32_t>((R - 1) / 2);
  }
  __syncthreads();
  for (int bb = sh.bytes64 - 1; bb >= 0; --bb) {
    for (int i = tid; i < 256; i += kSelThreads) sh.hist[i] = 0;
    __syncthreads();
    const int shift = 8 * bb;
    const int64_t lo = sh.lo64;
    const uint64_t pref = sh.pref64;
    for (int64_t r = tid; r < R; r += kSelThreads) {
      const uint64_t off = static_cast<uint64_t>(value(r) - lo);
      if (shift + 8 >= 64 || (off >> (shift + 8)) == (pref >> (shift + 8)))
        atomicAdd(&sh.hist[static_cast<uint32_t>(off >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (warp == 0) {
      uint32_t digit, below;
      hist_find(sh.hist, sh.rem, lane, digit, below);
      if (lane == 0) {
        sh.rem -= below;
        sh.pref64 |= static_cast<uint64_t>(digit) << shift;
      }
    }
    __syncthreads();
  }
  if (tid == 0) sh.med = sh.lo64 + static_cast<int64_t>(sh.pref64);
  __syncthreads();
}

// The first pass of a column's selection resolves kWideBits bits at once, in
// a 2^kWideBits-bin histogram that lives in the candidate slots (unused
// until the next pass).
constexpr int kWideBits = 11;
constexpr int kWideBins = 1 << kWideBits;
static_assert(kWideBins <= kSelCand, "the wide histogram lives in the candidate slots");

// The bin of a 2048-bin shared-memory histogram (16-byte aligned) that holds
// rank `rem`, and the count below it: each lane sums 64 consecutive bins, one
// warp scan picks the owning lane, and the owner's 64 bins are split two per
// lane for a second scan.  Whole warp; results in every lane.
__device__ __forceinline__ void hist_find_wide(const uint32_t* h, uint32_t rem, int lane, uint32_t& digit,
                                               uint32_t& below) {
  const uint4* h4 = reinterpret_cast<const uint4*>(h) + 16 * lane;
  uint32_t sum = 0;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const uint4 v = h4[j];
    sum += v.x + v.y + v.z + v.w;
  }
  uint32_t incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t up = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += up;
  }
  const uint32_t excl = incl - sum;
  const int owner = __ffs(__ballot_sync(kFull, excl <= rem && rem < incl)) - 1;
  const uint32_t base = __shfl_sync(kFull, excl, owner);
  const uint32_t r = rem - base;  // rank within the owner's 64 bins
  const uint2 pr = reinterpret_cast<const uint2*>(h + 64 * owner)[lane];
  const uint32_t two = pr.x + pr.y;
  uint32_t in2 = two;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t up = __shfl_up_sync(kFull, in2, o);
    if (lane >= o) in2 += up;
  }
  const uint32_t ex2 = in2 - two;
  const int sub = __ffs(__ballot_sync(kFull, ex2 <= r && r < in2)) - 1;
  const uint32_t e2 = __shfl_sync(kFull, ex2, sub);
  const uint32_t x = __shfl_sync(kFull, pr.x, sub);
  const bool second = r - e2 >= x;  // past the pair's first bin
  digit = 64u * owner + 2u * sub + (second ? 1u : 0u);
  below = base + e2 + (second ? x : 0u);
}

__global__ void __launch_bounds__(kSelThreads, kSelPerSM) rank_select_kernel(const RankParams p) {
  __shared__ __align__(16) SelShared sh;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int S = static_cast<int>(p.S);
  const int R = static_cast<int>(p.R);
  const int64_t tasks = p.Tc * S;
  // this chunk's encode (and, through its own wait, every earlier kernel) is
  // complete and visible; then the next chunk's encode may start
  griddep_wait();
  griddep_launch_dependents();
  for (int64_t task = blockIdx.x; task < tasks; task += gridDim.x) {
    const int64_t tl = task / S;
    const int s = static_cast<int>(task - tl * S);
    const int64_t t = p.c0 + tl;
    // ---- the column's key range, second largest and out-of-range flag from the encode blocks
    if (warp == 0) {
      uint32_t mn = 0xffffffffu, x1 = 0u, x2 = 0u, bad = 0u;
      for (int b = lane; b < p.nblk; b += 32) {
        const int64_t item = tl * p.nblk + b;
        mn = min(mn, p.pmin[item * S + s]);
        top2_merge<uint32_t>(x1, x2, p.pmax[item * S + s], p.psec[item * S + s]);
        bad |= p.pbad[item];
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const uint32_t o1 = __shfl_xor_sync(kFull, x1, o);
        const uint32_t o2 = __shfl_xor_sync(kFull, x2, o);
        top2_merge<uint32_t>(x1, x2, o1, o2);
      }
      mn = __reduce_min_sync(kFull, mn);
      bad = __reduce_or_sync(kFull, bad);
      if (lane == 0) {
        sh.lo = mn;
        sh.hi = x1;
        sh.sec_key = R >= 2 ? x2 : x1;
        sh.bad = bad;
        const uint32_t range = x1 - mn;
        sh.nb = range ? 32 - __clz(static_cast<int>(range)) : 0;
        sh.pref = 0;
        sh.rem = static_cast<uint32_t>((R - 1) / 2);
        sh.ncand = 0;
        sh.compact = 0;
      }
    }
    __syncthreads();
    const uint32_t* col = p.keys + (tl * S + s) * p.ldR;
    if (sh.bad) {
      select_column_64(p, t, s, sh);
    } else {
      const uint32_t lo = sh.lo;
      const int nb = sh.nb;
      // ---- first pass: every key counts; the top kWideBits bits of the range
      // go into the wide histogram (the candidate slots), four keys per load
      int start_hi = 0;  // bits still to resolve after the first pass
      if (nb > 0) {
        const int shift = nb > kWideBits ? nb - kWideBits : 0;  // offsets are below 2^nb
        uint32_t* wide = sh.cand;
        for (int i = tid; i < kWideBins / 4; i += kSelThreads)
          reinterpret_cast<uint4*>(wide)[i] = make_uint4(0, 0, 0, 0);
        __syncthreads();
        const int nq = R >> 2;
        for (int i = tid; i < nq; i += kSelThreads) {
          const uint4 k4 = reinterpret_cast<const uint4*>(col)[i];
          atomicAdd(&wide[((k4.x - lo) >> shift) & (kWideBins - 1)], 1u);
          atomicAdd(&wide[((k4.y - lo) >> shift) & (kWideBins - 1)], 1u);
          atomicAdd(&wide[((k4.z - lo) >> shift) & (kWideBins - 1)], 1u);
          atomicAdd(&wide[((k4.w - lo) >> shift) & (kWideBins - 1)], 1u);
        }
        for (int r = 4 * nq + tid; r < R; r += kSelThreads)
          atomicAdd(&wide[((col[r] - lo) >> shift) & (kWideBins - 1)], 1u);
        __syncthreads();
        if (warp == 0) {
          uint32_t digit, below;
          hist_find_wide(wide, sh.rem, lane, digit, below);
          if (lane == 0) {
            sh.pref = digit << shift;
            sh.rem -= below;
            sh.kept = wide[digit];
            sh.compact = shift > 0 && wide[digit] <= kSelCand;
          }
        }
        __syncthreads();
        start_hi = shift;
        if (shift > 0 && sh.kept <= 32) {
          // ---- at most 32 keys share the chosen bin: gather them (the
          // wide histogram is dead) and rank them by counting in one warp
          __syncthreads();  // every thread has read kept
          if (tid == 0) sh.ncand = 0;
          __syncthreads();
          const uint32_t dsel = sh.pref >> shift;
          auto gather = [&](uint32_t k) {
            if (((k - lo) >> shift) == dsel) sh.cand[atomicAdd(&sh.ncand, 1u)] = k - lo;
          };
          for (int i = tid; i < nq; i += kSelThreads) {
            const uint4 k4 = reinterpret_cast<const uint4*>(col)[i];
            gather(k4.x);
            gather(k4.y);
            gather(k4.z);
            gather(k4.w);
          }
          for (int r = 4 * nq + tid; r < R; r += kSelThreads) gather(col[r]);
          __syncthreads();
          if (warp == 0) {
            const uint32_t kept = sh.kept, rem = sh.rem;
            const uint32_t v = static_cast<uint32_t>(lane) < kept ? sh.cand[lane] : 0xffffffffu;
            uint32_t lt = 0, le = 0;
            for (uint32_t q = 0; q < kept; ++q) {
              const uint32_t c = __shfl_sync(kFull, v, static_cast<int>(q));
              lt += c < v ? 1u : 0u;
              le += c <= v ? 1u : 0u;
            }
            const uint32_t hit = __ballot_sync(kFull, static_cast<uint32_t>(lane) < kept && lt <= rem && rem < le);
            const uint32_t ans = __shfl_sync(kFull, v, __ffs(hit) - 1);
            if (lane == 0) sh.pref = ans;
          }
          start_hi = 0;
        }
      }
      // ---- later passes: 8 bits each below the top digit
      bool read_all = true;  // the column is still read from L2
      for (int hi = start_hi; hi > 0; hi -= 8) {
        const int shift = hi > 8 ? hi - 8 : 0;
        const uint32_t mask = (1u << (hi - shift)) - 1u;
        __syncthreads();  // the last digit search is done: its pref and rem are visible, hist is free
        const uint32_t pref = sh.pref;
        const bool compact = sh.compact != 0;
        for (int i = tid; i < 256; i += kSelThreads) sh.hist[i] = 0;
        __syncthreads();
        if (read_all) {
          // second pass: count the matching keys; keep them when they are few
          const int nq = R >> 2;
          for (int i = tid; i < nq + (R & 3); i += kSelThreads) {
            uint32_t k[4];
            int nk = 4;
            if (i < nq) {
              const uint4 k4 = reinterpret_cast<const uint4*>(col)[i];
              k[0] = k4.x;
              k[1] = k4.y;
              k[2] = k4.z;
              k[3] = k4.w;
            } else {
              k[0] = col[4 * nq + (i - nq)];
              nk = 1;
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              if (j >= nk) break;
              const uint32_t o = k[j] - lo;
              if (((o ^ pref) >> hi) == 0) {
                atomicAdd(&sh.hist[(o >> shift) & mask], 1u);
                if (compact) sh.cand[atomicAdd(&sh.ncand, 1u)] = k[j];
              }
            }
          }
          if (compact) read_all = false;
        } else {
          const int n = static_cast<int>(sh.ncand);
          for (int i = tid; i < n; i += kSelThreads) {
            const uint32_t o = sh.cand[i] - lo;
            if (((o ^ pref) >> hi) == 0) atomicAdd(&sh.hist[(o >> shift) & mask], 1u);
          }
        }
        __syncthreads();
        if (warp == 0) {
          uint32_t digit, below;
          hist_find(sh.hist, sh.rem, lane, digit, below);
          if (lane == 0) {
            sh.pref |= digit << shift;
            sh.rem -= below;
          }
        }
      }
      __syncthreads();
      if (tid == 0) {
        const int64_t ref = p.ref[tl * S + s];
        sh.med = key_value(ref, lo + sh.pref);
        sh.F = key_value(ref, sh.hi);
        sh.sec = key_value(ref, sh.sec_key);
      }
    }
    // the column's scratch is dead: drop its lines from L2 without write-back
    for (int off = tid * 32; off < p.ldR; off += kSelThreads * 32) discard_l2_line(col + off);
    __syncthreads();
    if (tid == 0) {
      const int64_t lag = sh.F - sh.med;
      if (p.of_prefix) {
        const int64_t gap = sh.F - sh.sec;
        if (p.L) p.L[t * S + s] = lag;
        if (p.G) p.G[t * S + s] = gap;
        const int64_t w = (p.t0 + t) / p.W - p.w_first;
        if (p.Lw && lag)
          atomicAdd(reinterpret_cast<unsigned long long*>(&p.Lw[w * S + s]), static_cast<unsigned long long>(lag));
        if (p.Gw && gap)
          atomicAdd(reinterpret_cast<unsigned long long*>(&p.Gw[w * S + s]), static_cast<unsigned long long>(gap));
      } else {
        const int64_t w = (p.t0 + t) / p.W - p.w_first;
        if (lag) atomicAdd(reinterpret_cast<unsigned long long*>(&p.spread[w * S + s]),
                           static_cast<unsigned long long>(lag));
      }
    }
    __syncthreads();  // sh is rewritten by the next task
  }
}

// Delta-lag per step row, one thread per step: dL[s] = L[s] - L[s-1],
// L[-1] = 0.  Walking s downwards lets dL alias L (in-place conversion).
__global__ void lag_delta_kernel(const int64_t* L, int64_t T, int S, int64_t* dL) {
  for (int64_t t = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; t < T; t += int64_t(gridDim.x) * blockDim.x) {
    const int64_t* l = L + t * S;
    int64_t* o = dL + t * S;
    for (int s = S - 1; s > 0; --s) o[s] = l[s] - l[s - 1];
    o[0] = l[0];
  }
}

struct ScratchLayout {
  int64_t ldR;
  int nblk;
  size_t keys, pmin, pmax, psec, pbad, ref, total;  // byte offsets within the workspace
};

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

ScratchLayout layout_for(int64_t R, int64_t S, int64_t Tc) {
  ScratchLayout l{};
  l.ldR = (R + 31) & ~int64_t(31);
  l.nblk = static_cast<int>((R + kEncRows - 1) / kEncRows);
  size_t at = 0;
  l.keys = at;
  at = align256(at + size_t(Tc) * S * l.ldR * 4);
  l.pmin = at;
  at = align256(at + size_t(Tc) * l.nblk * S * 4);
  l.pmax = at;
  at = align256(at + size_t(Tc) * l.nblk * S * 4);
  l.psec = at;
  at = align256(at + size_t(Tc) * l.nblk * S * 4);
  l.pbad = at;
  at = align256(at + size_t(Tc) * l.nblk * 4);
  l.ref = at;
  at = align256(at + size_t(Tc) * S * 8);
  l.total = at;
  return l;
}

// steps per chunk that `bytes` of scratch holds (0: not even one)
int64_t chunk_steps_for(int64_t T, int64_t R, int64_t S, size_t bytes) {
  if (layout_for(R, S, 1).total > bytes) return 0;
  int64_t lo = 1, hi = T;
  while (lo < hi) {
    const int64_t mid = lo + (hi - lo + 1) / 2;
    if (layout_for(R, S, mid).total <= bytes)
      lo = mid;
    else
      hi = mid - 1;
  }
  return lo;
}

template <typename K>
cudaError_t launch_pdl(K kern, int grid, int threads, const RankParams& p, cudaStream_t stream, bool overlap = true) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = overlap ? 1 : 0;
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(static_cast<unsigned>(threads));
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, p);
}

// first: the call's first chunk.  Its encode starts only once everything
// before it on the stream has completed: the previous call's last select may
// still be reading the same scratch buffer.
template <int SC>
cudaError_t launch_encode(const RankParams& p, cudaStream_t stream, bool first) {
  // the split-row kernel for 4, 8 and 16 stages, the row-per-thread one otherwise
  constexpr bool kSplit = SC == 4 || SC == 8 || SC == 16;
  auto kern = kSplit ? rank_encode_split_kernel<kSplit ? SC : 8> : rank_encode_kernel<SC>;
  static int per_sm = 0;  // resident CTAs per SM (same on every GB300)
  if (per_sm == 0 &&
      (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kEncThreads, 0) != cudaSuccess || per_sm < 1)) {
    cudaGetLastError();
    per_sm = 1;
  }
  const int grid = static_cast<int>(std::min<int64_t>(p.Tc * p.nblk, int64_t(per_sm) * sm_count()));
  return launch_pdl(kern, grid, kEncThreads, p, stream, !first);
}

}  // namespace

// The workspace holds two chunk buffers: the encode of chunk c+1 fills one
// while the select of chunk c reads the other.
size_t rank_workspace_size(int64_t T, int64_t R, int64_t S) {
  if (T < 1 || R < 1 || S < 1) return 0;
  const size_t one = layout_for(R, S, 1).total;
  const int64_t want = std::max<int64_t>(1, std::min<int64_t>(T, int64_t(kRkChunkTarget / one)));
  return 2 * layout_for(R, S, want).total;
}

bool rank_workspace_ok(int64_t T, int64_t R, int64_t S, size_t bytes) {
  return chunk_steps_for(T, R, S, bytes / 2 & ~size_t(255)) > 0;
}

cudaError_t launch_rank_select(const int64_t* d, int64_t T, int64_t R, int64_t S, int of_prefix, int64_t t0,
                               int64_t W, int64_t* L, int64_t* dL, int64_t* G, int64_t* Lw, int64_t* Gw,
                               int64_t* spread, void* workspace, size_t ws_bytes, uint32_t* status,
                               cudaStream_t stream) {
  const size_t half = ws_bytes / 2 & ~size_t(255);  // one chunk buffer, 256-byte aligned
  const int64_t Tc = chunk_steps_for(T, R, S, half);
  if (Tc < 1) return cudaErrorInvalidValue;
  const ScratchLayout l = layout_for(R, S, Tc);
  unsigned char* const ws_base = static_cast<unsigned char*>(workspace);
  unsigned char* ws = ws_base;
  RankParams p{};
  p.d = d;
  p.T = T;
  p.R = R;
  p.S = S;
  p.of_prefix = of_prefix;
  p.t0 = t0;
  p.W = W;
  p.w_first = t0 / W;
  p.L = L ? L : dL;  // without L, the lag is written into dL and converted there
  p.G = G;
  p.Lw = Lw;
  p.Gw = Gw;
  p.spread = spread;
  p.status = status;
  p.ldR = l.ldR;
  p.nblk = l.nblk;
  p.keys = reinterpret_cast<uint32_t*>(ws + l.keys);
  p.pmin = reinterpret_cast<uint32_t*>(ws + l.pmin);
  p.pmax = reinterpret_cast<uint32_t*>(ws + l.pmax);
  p.psec = reinterpret_cast<uint32_t*>(ws + l.psec);
  p.pbad = reinterpret_cast<uint32_t*>(ws + l.pbad);
  p.ref = reinterpret_cast<int64_t*>(ws + l.ref);
  const int sms = sm_count();
  for (int64_t c0 = 0, c = 0; c0 < T; c0 += Tc, ++c) {
    p.c0 = c0;
    p.Tc = std::min(Tc, T - c0);
    ws = ws_base + (c & 1) * half;  // alternate the two chunk buffers
    p.keys = reinterpret_cast<uint32_t*>(ws + l.keys);
    p.pmin = reinterpret_cast<uint32_t*>(ws + l.pmin);
    p.pmax = reinterpret_cast<uint32_t*>(ws + l.pmax);
    p.psec = reinterpret_cast<uint32_t*>(ws + l.psec);
    p.pbad = reinterpret_cast<uint32_t*>(ws + l.pbad);
    p.ref = reinterpret_cast<int64_t*>(ws + l.ref);
    count_launch();
    cudaError_t e;
    switch (S) {
      case 4: e = launch_encode<4>(p, stream, c == 0); break;
      case 6: e = launch_encode<6>(p, stream, c == 0); break;
      case 8: e = launch_encode<8>(p, stream, c == 0); break;
      case 10: e = launch_encode<10>(p, stream, c == 0); break;
      case 16: e = launch_encode<16>(p, stream, c == 0); break;
      default: e = launch_encode<0>(p, stream, c == 0); break;
    }
    if (e != cudaSuccess) return e;
    const int sel_grid = static_cast<int>(std::min<int64_t>(p.Tc * S, int64_t(sms) * kSelPerSM));
    count_launch();
    if ((e = launch_pdl(rank_select_kernel, sel_grid, kSelThreads, p, stream)) != cudaSuccess) return e;
  }
  if (of_prefix && dL) {
    const int grid = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>((T + 255) / 256, int64_t(sms) * 4)));
    count_launch();
    lag_delta_kernel<<<grid, 256, 0, stream>>>(p.L, T, static_cast<int>(S), dL);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace sf

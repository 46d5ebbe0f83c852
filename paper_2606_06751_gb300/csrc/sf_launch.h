// sf_launch.h - host-side interface between the C ABI layer (sf_api.cu) and
// the kernel translation units.  Internal to libstagefrontier.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "stagefrontier.h"

namespace sf {

// Everything a streaming pass over d needs; unused outputs are null.
struct StreamJob {
  const int64_t* d = nullptr;
  int64_t T = 0, R = 0, S = 0;
  // sf_frontier outputs
  int64_t* a = nullptr;
  int32_t* lead = nullptr;
  int64_t* mk = nullptr;
  // sf_window_aggregate outputs (and the evidence pass's X / D)
  int64_t* X = nullptr;
  int64_t* D = nullptr;
  int64_t* E = nullptr;
  int32_t* C = nullptr;
  uint8_t* step_lead = nullptr;
  int64_t t0 = 0, W = 1;
  // evidence pass (sf_direct_gain)
  bool gain = false;
  const int64_t* m = nullptr;
  const int64_t* wall = nullptr;
  int32_t other_stage = -1;
  int64_t eta_num = 0, eta_den = 1;
  int64_t* Y = nullptr;
  uint64_t* quality = nullptr;
  uint32_t* status = nullptr;
  // routing-baseline pass (sf_window_baselines)
  bool base = false;
  // the previous launch on the stream is this call's clear of its outputs
  // (launch_zero_many): the pass is launched as its programmatic dependent,
  // streaming its first tiles while the clear runs, and writes nothing
  // before that clear has completed
  bool after_clear = false;
  int64_t* bM = nullptr;
  uint64_t* bSUM = nullptr;
  int64_t* bSLOW = nullptr;
  int64_t* bRANK0 = nullptr;
};

// cuTensorMapEncodeTiled from the driver, resolved once (null if unavailable).
using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                              CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                              CUtensorMapFloatOOBfill);
EncodeFn encode_fn();

int sm_count();                     // SMs of the current device (cached)
void count_launch(uint64_t n = 1);  // bump the library's launch counter

cudaError_t launch_zero(void* p, size_t bytes, cudaStream_t stream);
// Up to kZeroMax buffers (whole 4-byte words) cleared by one launch; null or empty entries are skipped.
constexpr int kZeroMax = 6;
struct ZeroList {
  void* ptr[kZeroMax];
  size_t words[kZeroMax];
  int n = 0;
  void add(void* p, size_t bytes) {
    if (p && bytes) {
      ptr[n] = p;
      words[n] = bytes / 4;
      ++n;
    }
  }
};
// *launched (when given) tells whether a kernel was enqueued: nothing is when
// every entry is empty.  The clear lets the next launch on the stream start
// early (programmatic dependent launch, StreamJob::after_clear).
cudaError_t launch_zero_many(const ZeroList& z, cudaStream_t stream, bool* launched = nullptr);
cudaError_t launch_wait_selftest(uint64_t limit_ns, uint32_t* status, cudaStream_t stream);
cudaError_t launch_stream_pass(const StreamJob& job, cudaStream_t stream);
// ties[t,s] = number of ranks whose prefix equals F[t,s] (F rebuilt from the increments a)
cudaError_t launch_frontier_ties(const int64_t* d, int64_t T, int64_t R, int64_t S, const int64_t* a,
                                 int32_t* ties, uint32_t* status, cudaStream_t stream);
cudaError_t launch_window_median(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W,
                                 int64_t* m, uint32_t* status, cudaStream_t stream);
cudaError_t launch_rank_select(const int64_t* d, int64_t T, int64_t R, int64_t S, int of_prefix, int64_t t0,
                               int64_t W, int64_t* L, int64_t* dL, int64_t* G, int64_t* Lw, int64_t* Gw,
                               int64_t* spread, void* workspace, size_t ws_bytes, uint32_t* status,
                               cudaStream_t stream);
size_t rank_workspace_size(int64_t T, int64_t R, int64_t S);
bool rank_workspace_ok(int64_t T, int64_t R, int64_t S, size_t bytes);
cudaError_t launch_group_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, const int32_t* group, int64_t G,
                                 int64_t t0, int64_t W, int64_t* Xg, int64_t* Dg, uint32_t* status,
                                 cudaStream_t stream);
cudaError_t launch_stage_group_sum(const int64_t* X, int64_t nW, int64_t S, const int32_t* stage_group, int64_t K,
                                   int64_t* Y, cudaStream_t stream);
cudaError_t launch_gathered_to_steps(const int64_t* src, int64_t T, int64_t R, int64_t S, int64_t N, int64_t* dst,
                                     cudaStream_t stream);
cudaError_t launch_topk(const int64_t* X, const int64_t* E, int64_t nW, int64_t S, int64_t R,
                        int32_t k, int32_t* top_stage, int64_t* top_stage_value, int32_t* top_pair,
                        int64_t* top_pair_value, cudaStream_t stream);

struct GateJob {
  int64_t T, R, S, W, nW;
  const int64_t *X, *Y, *D;
  const uint8_t* step_lead;
  const uint64_t* quality;
  const int32_t* role;
  const int32_t* missing;
  sf_label_config cfg;
  uint32_t *labels, *route_mask, *amb_mask;
  double *share, *gain;
  int32_t *n_confident, *n_switch;
};
cudaError_t launch_gates(const GateJob& job, cudaStream_t stream);

}  // namespace sf

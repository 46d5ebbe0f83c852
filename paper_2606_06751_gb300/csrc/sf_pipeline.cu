// sf_pipeline.cu - sf_stream_windows: the whole hot path over a telemetry
// tensor that lives in HOST memory.  The tensor is cut into chunks of whole
// windows; each chunk is copied host->device on the copy stream into one of
// two caller-provided device staging buffers, then the compute stream runs the
// window medians, the fused evidence pass (frontier, aggregates, lead-rank
// credit, gain numerators), top-k suspects and the gates on it, writing the
// chunk's windows into the caller's output rows.  The copy of chunk c+1 runs
// while chunk c is computed; a staging buffer is refilled only after the
// compute stream has finished with it.  Host code only: every computation is
// a kernel launched through the other entry points.
#include <algorithm>

#include "sf_launch.h"
#include "stagefrontier.h"

namespace {

struct Events {
  cudaEvent_t copied[2] = {nullptr, nullptr};  // chunk in buffer b has landed
  cudaEvent_t freed[2] = {nullptr, nullptr};   // compute has finished with buffer b
  ~Events() {
    for (int b = 0; b < 2; ++b) {
      if (copied[b]) cudaEventDestroy(copied[b]);
      if (freed[b]) cudaEventDestroy(freed[b]);
    }
  }
  bool create() {
    for (int b = 0; b < 2; ++b)
      if (cudaEventCreateWithFlags(&copied[b], cudaEventDisableTiming) != cudaSuccess ||
          cudaEventCreateWithFlags(&freed[b], cudaEventDisableTiming) != cudaSuccess)
        return false;
    return true;
  }
};

// gathered = false: h_d is [T][R][S]; true: h_d holds the windows' gathered
// [R][n][S] blocks one after another, converted on the device after the copy.
sf_status stream_windows(bool gathered, const int64_t* h_d, int64_t T, int64_t R, int64_t S, int64_t W, int32_t k,
                         int64_t chunk_steps, const sf_label_config* cfg, int64_t* staging, size_t staging_bytes,
                         void* workspace, size_t workspace_bytes, int64_t* X, int64_t* Y, int64_t* D, int64_t* E,
                         int32_t* C, int32_t* top_stage, int32_t* top_pair, int64_t* top_pair_value,
                         uint32_t* labels, uint32_t* route_mask, uint32_t* amb_mask, double* share, double* gain,
                         uint32_t* status, cudaStream_t stream, cudaStream_t copy_stream) {
  if (!h_d || !cfg || !staging || !X || !Y || !D || !labels || !route_mask || !amb_mask || T < 1 || R < 1 ||
      R > 65536 || S < 1 || S > 32 || W < 1 || W > 65536 || k < 1 || k > 32 || chunk_steps < 1 ||
      chunk_steps % W != 0 || T > (int64_t(1) << 62) / (R * S))
    return SF_EINVAL;
  if (reinterpret_cast<uintptr_t>(h_d) % 16 != 0 || reinterpret_cast<uintptr_t>(staging) % 16 != 0)
    return SF_EINVAL_ALIGN;
  const int64_t chunk = std::min(chunk_steps, T);
  const size_t chunk_bytes = size_t(chunk) * R * S * 8;
  const size_t buf_bytes = (chunk_bytes + 255) & ~size_t(255);  // second buffer 256-byte aligned
  if (staging_bytes < (gathered ? 3 : 2) * buf_bytes) return SF_EWORKSPACE;
  const int64_t nW_chunk = (chunk + W - 1) / W;
  const size_t need = sf_label_windows_workspace_size(chunk, R, S, W);
  if (!workspace || workspace_bytes < need) return SF_EWORKSPACE;
  Events ev;
  if (!ev.create()) return SF_ECUDA;
  int64_t* buf[2] = {staging, reinterpret_cast<int64_t*>(reinterpret_cast<unsigned char*>(staging) + buf_bytes)};
  // gathered input: the chunk converted to [n][R][S] for the kernels
  int64_t* steps_buf = reinterpret_cast<int64_t*>(reinterpret_cast<unsigned char*>(staging) + 2 * buf_bytes);
  // workspace carve-up of one chunk's labeler: medians, step leaders, quality (unused here)
  unsigned char* ws = static_cast<unsigned char*>(workspace);
  int64_t* m = reinterpret_cast<int64_t*>(ws);
  uint8_t* sl = ws + ((size_t(nW_chunk) * R * S * 8 + 255) & ~size_t(255));
  if (size_t(nW_chunk) * R * S * 8 + 256 + size_t(chunk) > workspace_bytes) return SF_EWORKSPACE;

  const int64_t nchunks = (T + chunk - 1) / chunk;
  for (int64_t c = 0; c < nchunks; ++c) {
    const int b = static_cast<int>(c & 1);
    const int64_t t0 = c * chunk, n = std::min(chunk, T - t0), w0 = t0 / W;
    // refill buffer b only after the compute stream is done with chunk c-2
    if (c >= 2 && cudaStreamWaitEvent(copy_stream, ev.freed[b], 0) != cudaSuccess) return SF_ECUDA;
    if (cudaMemcpyAsync(buf[b], h_d + t0 * R * S, size_t(n) * R * S * 8, cudaMemcpyHostToDevice, copy_stream) !=
            cudaSuccess ||
        cudaEventRecord(ev.copied[b], copy_stream) != cudaSuccess ||
        cudaStreamWaitEvent(stream, ev.copied[b], 0) != cudaSuccess)
      return SF_ECUDA;
    const int64_t nW = (n + W - 1) / W;
    const int64_t* dc = buf[b];
    if (gathered) {
      // the chunk's windows are whole gathered blocks of W steps (the last may be short)
      if (sf::launch_gathered_to_steps(buf[b], n, R, S, W, steps_buf, stream) != cudaSuccess ||
          cudaEventRecord(ev.freed[b], stream) != cudaSuccess)
        return SF_ECUDA;
      dc = steps_buf;
    }
    sf_status st = sf_window_median(dc, n, R, S, W, m, status, stream);
    if (st == SF_OK)
      st = sf_direct_gain(dc, n, R, S, W, m, nullptr, -1, cfg->eta_Q, X + w0 * S, Y + w0 * S, D + w0,
                          E ? E + w0 * S * R : nullptr, C ? C + w0 * S * R : nullptr, sl, nullptr, status, stream);
    if (st == SF_OK && (top_stage || top_pair || top_pair_value))
      st = sf_topk_suspects(X + w0 * S, E ? E + w0 * S * R : nullptr, nW, S, R, k,
                            top_stage ? top_stage + w0 * k : nullptr, nullptr,
                            (E && top_pair) ? top_pair + w0 * k * 2 : nullptr,
                            (E && top_pair_value) ? top_pair_value + w0 * k : nullptr, stream);
    if (st == SF_OK)
      st = sf_label_gates(n, R, S, W, X + w0 * S, Y + w0 * S, D + w0, sl, nullptr, nullptr, nullptr, cfg,
                          labels + w0, route_mask + w0, amb_mask + w0, share ? share + w0 * S : nullptr,
                          gain ? gain + w0 * S : nullptr, nullptr, nullptr, stream);
    if (st != SF_OK) return st;
    if (!gathered && cudaEventRecord(ev.freed[b], stream) != cudaSuccess) return SF_ECUDA;
  }
  // the events are destroyed on return; pending work still completes in order
  return SF_OK;
}

}  // namespace

extern "C" sf_status sf_stream_windows(const int64_t* h_d, int64_t T, int64_t R, int64_t S, int64_t W, int32_t k,
                                       int64_t chunk_steps, const sf_label_config* cfg, int64_t* staging,
                                       size_t staging_bytes, void* workspace, size_t workspace_bytes,
                                       int64_t* X, int64_t* Y, int64_t* D, int64_t* E, int32_t* C,
                                       int32_t* top_stage, int32_t* top_pair, int64_t* top_pair_value,
                                       uint32_t* labels, uint32_t* route_mask, uint32_t* amb_mask, double* share,
                                       double* gain, uint32_t* status, cudaStream_t stream,
                                       cudaStream_t copy_stream) {
  return stream_windows(false, h_d, T, R, S, W, k, chunk_steps, cfg, staging, staging_bytes, workspace,
                        workspace_bytes, X, Y, D, E, C, top_stage, top_pair, top_pair_value, labels, route_mask,
                        amb_mask, share, gain, status, stream, copy_stream);
}

extern "C" sf_status sf_stream_gathered_windows(const int64_t* h_g, int64_t T, int64_t R, int64_t S, int64_t W,
                                                int32_t k, int64_t chunk_steps, const sf_label_config* cfg,
                                                int64_t* staging, size_t staging_bytes, void* workspace,
                                                size_t workspace_bytes, int64_t* X, int64_t* Y, int64_t* D,
                                                int64_t* E, int32_t* C, int32_t* top_stage, int32_t* top_pair,
                                                int64_t* top_pair_value, uint32_t* labels, uint32_t* route_mask,
                                                uint32_t* amb_mask, double* share, double* gain, uint32_t* status,
                                                cudaStream_t stream, cudaStream_t copy_stream) {
  return stream_windows(true, h_g, T, R, S, W, k, chunk_steps, cfg, staging, staging_bytes, workspace,
                        workspace_bytes, X, Y, D, E, C, top_stage, top_pair, top_pair_value, labels, route_mask,
                        amb_mask, share, gain, status, stream, copy_stream);
}

extern "C" size_t sf_stream_windows_staging_size(int64_t T, int64_t R, int64_t S, int64_t chunk_steps) {
  if (T < 1 || R < 1 || S < 1 || chunk_steps < 1) return 0;
  const size_t chunk_bytes = size_t(std::min(chunk_steps, T)) * R * S * 8;
  return 2 * ((chunk_bytes + 255) & ~size_t(255));
}

extern "C" size_t sf_stream_gathered_staging_size(int64_t T, int64_t R, int64_t S, int64_t chunk_steps) {
  if (T < 1 || R < 1 || S < 1 || chunk_steps < 1) return 0;
  const size_t chunk_bytes = size_t(std::min(chunk_steps, T)) * R * S * 8;
  return 3 * ((chunk_bytes + 255) & ~size_t(255));
}

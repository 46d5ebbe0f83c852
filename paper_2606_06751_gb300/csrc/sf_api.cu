// sf_api.cu - the C ABI of libstagefrontier (declared in stagefrontier.h):
// argument validation, output clearing, workspace carving and launch
// sequencing.  Every computation happens in the kernels (sf_stream.cu,
// sf_select.cu, sf_rank.cu, sf_group.cu, sf_ingest.cu); this file performs no
// arithmetic on the data.
#include <atomic>
#include <cstring>

#include "sf_device.cuh"
#include "sf_launch.h"
#include "stagefrontier.h"

namespace sf {

namespace {
std::atomic<uint64_t> g_launches{0};
constexpr int kMaxDevices = 64;
std::atomic<int> g_sms[kMaxDevices];

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

bool shape_ok(int64_t T, int64_t R, int64_t S) {
  if (T < 1 || R < 1 || R > 65536 || S < 1 || S > 32) return false;
  return T <= (int64_t(1) << 62) / (R * S);  // T*R*S*8 fits int64
}

bool ratio_ok(sf_ratio r) {
  return r.den > 0 && r.den <= (int64_t(1) << 31) && r.num >= 0 && r.num <= (int64_t(1) << 31);
}

bool config_ok(const sf_label_config* c) {
  return c && ratio_ok(c->gamma_A) && ratio_ok(c->gamma_G) && ratio_ok(c->eta_A) && ratio_ok(c->eta_G) &&
         ratio_ok(c->tau_C) && ratio_ok(c->eta_Q) && ratio_ok(c->gamma_switch) && ratio_ok(c->gamma_elig) &&
         ratio_ok(c->closure_max) && ratio_ok(c->overlap_max);
}

sf_status cuda_status(cudaError_t e) { return e == cudaSuccess ? SF_OK : SF_ECUDA; }

size_t round256(size_t x) { return (x + 255) & ~size_t(255); }

struct LabelLayout {
  size_t m, X, Y, D, q, sl, total;
};

LabelLayout label_layout(int64_t T, int64_t R, int64_t S, int64_t W) {
  const int64_t nW = (T + W - 1) / W;
  LabelLayout L{};
  size_t off = 0;
  L.m = off;
  off += round256(size_t(nW) * R * S * 8);
  L.X = off;
  off += round256(size_t(nW) * S * 8);
  L.Y = off;
  off += round256(size_t(nW) * S * 8);
  L.D = off;
  off += round256(size_t(nW) * 8);
  L.q = off;
  off += round256(size_t(nW) * 6 * 8);
  L.sl = off;
  off += round256(size_t(T));
  L.total = off;
  return L;
}
}  // namespace

int sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 1;
  int v = g_sms[dev].load(std::memory_order_relaxed);
  if (v <= 0) {
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) v = 1;
    g_sms[dev].store(v, std::memory_order_relaxed);
  }
  return v;
}

void count_launch(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

}  // namespace sf

using namespace sf;

extern "C" {

const char* sf_status_str(int code) {
  switch (code) {
    case SF_OK: return "ok";
    case SF_EINVAL: return "invalid argument";
    case SF_EINVAL_ALIGN: return "misaligned pointer";
    case SF_EUNSUPPORTED: return "unsupported shape";
    case SF_ECUDA: return "CUDA runtime error";
    case SF_EWORKSPACE: return "workspace missing or too small";
    default: return "unknown status";
  }
}

int64_t sf_num_windows(int64_t t0, int64_t T, int64_t W) {
  if (t0 < 0 || T < 1 || W < 1) return 0;
  return (t0 + T - 1) / W - t0 / W + 1;
}

uint64_t sf_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

void sf_label_config_default(sf_label_config* c) {
  if (!c) return;
  c->gamma_A = {2, 5};
  c->gamma_G = {1, 10};
  c->eta_A = {1, 20};
  c->eta_G = {1, 20};
  c->tau_C = {4, 5};
  c->eta_Q = {1, 20};
  c->gamma_switch = {1, 4};
  c->gamma_elig = {1, 2};
  c->closure_max = {1, 20};
  c->overlap_max = {1, 100};
  c->denom_floor_ns = 1;
  c->max_missing_ranks = 0;
  c->model_fit_mask = 0;
}

sf_status sf_frontier(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t* a, int32_t* lead,
                      int64_t* makespan, uint32_t* status, cudaStream_t stream) {
  if (!d || !shape_ok(T, R, S) || (!a && !lead && !makespan)) return SF_EINVAL;
  if (!aligned(d, 16) || !aligned(a, 8) || !aligned(lead, 4) || !aligned(makespan, 8) || !aligned(status, 4))
    return SF_EINVAL_ALIGN;
  StreamJob j;
  j.d = d;
  j.T = T;
  j.R = R;
  j.S = S;
  j.a = a;
  j.lead = lead;
  j.mk = makespan;
  j.status = status;
  return cuda_status(launch_stream_pass(j, stream));
}

sf_status sf_frontier_ties(const int64_t* d, int64_t T, int64_t R, int64_t S, const int64_t* a, int32_t* ties,
                           uint32_t* status, cudaStream_t stream) {
  if (!d || !a || !ties || !shape_ok(T, R, S)) return SF_EINVAL;
  if (!aligned(d, 16) || !aligned(a, 8) || !aligned(ties, 4) || !aligned(status, 4)) return SF_EINVAL_ALIGN;
  return cuda_status(launch_frontier_ties(d, T, R, S, a, ties, status, stream));
}

sf_status sf_window_aggregate(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W,
                              int64_t* X, int64_t* D, int64_t* E, int32_t* C, uint8_t* step_lead,
                              int32_t accumulate, uint32_t* status, cudaStream_t stream) {
  if (!d || !X || !D || !shape_ok(T, R, S) || t0 < 0 || W < 1 || W > 65536 ||
      (accumulate != 0 && accumulate != 1) || t0 > (int64_t(1) << 62) - T)
    return SF_EINVAL;
  if (!aligned(d, 16) || !aligned(X, 8) || !aligned(D, 8) || !aligned(E, 8) || !aligned(C, 4) ||
      !aligned(status, 4))
    return SF_EINVAL_ALIGN;
  const int64_t nW = sf_num_windows(t0, T, W);
  bool cleared = false;
  if (!accumulate) {
    ZeroList z;
    z.add(X, size_t(nW) * S * 8);
    z.add(D, size_t(nW) * 8);
    z.add(E, size_t(nW) * S * R * 8);
    z.add(C, size_t(nW) * S * R * 4);
    cudaError_t e = launch_zero_many(z, stream, &cleared);
    if (e != cudaSuccess) return SF_ECUDA;
  }
  StreamJob j;
  j.after_clear = cleared;
  j.d = d;
  j.T = T;
  j.R = R;
  j.S = S;
  j.X = X;
  j.D = D;
  j.E = E;
  j.C = C;
  j.step_lead = step_lead;
  j.t0 = t0;
  j.W = W;
  j.status = status;
  return cuda_status(launch_stream_pass(j, stream));
}

sf_status sf_window_baselines(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W,
                              int64_t* M, uint64_t* SUM, int64_t* SLOW, int64_t* RANK0, int32_t accumulate,
                              uint32_t* status, cudaStream_t stream) {
  if (!d || !M || !SUM || !SLOW || !RANK0 || !shape_ok(T, R, S) || t0 < 0 || W < 1 || W > 65536 ||
      (accumulate != 0 && accumulate != 1) || t0 > (int64_t(1) << 62) - T)
    return SF_EINVAL;
  if (!aligned(d, 16) || !aligned(M, 8) || !aligned(SUM, 8) || !aligned(SLOW, 8) || !aligned(RANK0, 8) ||
      !aligned(status, 4))
    return SF_EINVAL_ALIGN;
  const int64_t nW = sf_num_windows(t0, T, W);
  bool cleared = false;
  if (!accumulate) {
    ZeroList z;
    z.add(M, size_t(nW) * S * 8);
    z.add(SUM, size_t(nW) * S * 16);
    z.add(SLOW, size_t(nW) * S * 8);
    z.add(RANK0, size_t(nW) * S * 8);
    cudaError_t e = launch_zero_many(z, stream, &cleared);
    if (e != cudaSuccess) return SF_ECUDA;
  }
  StreamJob j;
  j.after_clear = cleared;
  j.d = d;
  j.T = T;
  j.R = R;
  j.S = S;
  j.t0 = t0;
  j.W = W;
  j.base = true;
  j.bM = M;
  j.bSUM = SUM;
  j.bSLOW = SLOW;
  j.bRANK0 = RANK0;
  j.status = status;
  return cuda_status(launch_stream_pass(j, stream));
}

sf_status sf_rank_lag(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t* L, int64_t* dL, int64_t* G,
                      void* workspace, size_t workspace_bytes, uint32_t* status, cudaStream_t stream) {
  if (!d || !shape_ok(T, R, S) || (!L && !dL && !G)) return SF_EINVAL;
  if (!aligned(d, 16) || !aligned(L, 8) || !aligned(dL, 8) || !aligned(G, 8) || !aligned(status, 4) ||
      !aligned(workspace, 256))
    return SF_EINVAL_ALIGN;
  if (!workspace || !rank_workspace_ok(T, R, S, workspace_bytes)) return SF_EWORKSPACE;
  return cuda_status(
      launch_rank_select(d, T, R, S, 1, 0, 1, L, dL, G, nullptr, nullptr, nullptr, workspace, workspace_bytes,
                         status, stream));
}

sf_status sf_raw_spread(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W, int64_t* spread,
                        int32_t accumulate, void* workspace, size_t workspace_bytes, uint32_t* status,
                        cudaStream_t stream) {
  if (!d || !spread || !shape_ok(T, R, S) || t0 < 0 || W < 1 || W > 65536 || (accumulate != 0 && accumulate != 1) ||
      t0 > (int64_t(1) << 62) - T)
    return SF_EINVAL;
  if (!aligned(d, 16) || !aligned(spread, 8) || !aligned(status, 4) || !aligned(workspace, 256))
    return SF_EINVAL_ALIGN;
  if (!workspace || !rank_workspace_ok(T, R, S, workspace_bytes)) return SF_EWORKSPACE;
  if (!accumulate && launch_zero(spread, size_t(sf_num_windows(t0, T, W)) * S * 8, stream) != cudaSuccess)
    return SF_ECUDA;
  return cuda_status(launch_rank_select(d, T, R, S, 0, t0, W, nullptr, nullptr, nullptr, nullptr, nullptr, spread,
                                        workspace, workspace_bytes, status, stream));
}

sf_status sf_rank_lag_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W,
                              int64_t* Lw, int64_t* Gw, int32_t accumulate, void* workspace, size_t workspace_bytes,
                              uint32_t* status, cudaStream_t stream) {
  if (!d || (!Lw && !Gw) || !shape_ok(T, R, S) || t0 < 0 || W < 1 || W > 65536 ||
      (accumulate != 0 && accumulate != 1) || t0 > (int64_t(1) << 62) - T)
    return SF_EINVAL;
  if (!aligned(d, 16) || !aligned(Lw, 8) || !aligned(Gw, 8) || !aligned(status, 4) || !aligned(workspace, 256))
    return SF_EINVAL_ALIGN;
  if (!workspace || !rank_workspace_ok(T, R, S, workspace_bytes)) return SF_EWORKSPACE;
  const size_t bytes = size_t(sf_num_windows(t0, T, W)) * S * 8;
  ZeroList z;
  z.add(Lw, bytes);
  z.add(Gw, bytes);
  if (!accumulate && launch_zero_many(z, stream) != cudaSuccess)
    return SF_ECUDA;
  return cuda_status(launch_rank_select(d, T, R, S, 1, t0, W, nullptr, nullptr, nullptr, Lw, Gw, nullptr, workspace,
                                        workspace_bytes, status, stream));
}

size_t sf_rank_workspace_size(int64_t T, int64_t R, int64_t S) {
  return shape_ok(T, R, S) ? rank_workspace_size(T, R, S) : 0;
}

sf_status sf_group_aggregate(const int64_t* d, int64_t T, int64_t R, int64_t S, const int32_t* group, int64_t G,
                             int64_t t0, int64_t W, int64_t* Xg, int64_t* Dg, int32_t accumulate, uint32_t* status,
                             cudaStream_t stream) {
  if (!d || !group || !Xg || !Dg || !shape_ok(T, R, S) || G < 1 || G > 4096 || G * S > 4096 || t0 < 0 || W < 1 ||
      W > 65536 || (accumulate != 0 && accumulate != 1) || t0 > (int64_t(1) << 62) - T)
    return SF_EINVAL;
  if (!aligned(d, 16) || !aligned(group, 4) || !aligned(Xg, 8) || !aligned(Dg, 8) || !aligned(status, 4))
    return SF_EINVAL_ALIGN;
  const size_t nW = size_t(sf_num_windows(t0, T, W));
  ZeroList z;
  z.add(Xg, nW * G * S * 8);
  z.add(Dg, nW * G * 8);
  if (!accumulate && launch_zero_many(z, stream) != cudaSuccess)
    return SF_ECUDA;
  return cuda_status(launch_group_windows(d, T, R, S, group, G, t0, W, Xg, Dg, status, stream));
}

sf_status sf_stage_group_sum(const int64_t* X, int64_t nW, int64_t S, const int32_t* stage_group, int64_t K,
                             int64_t* Y, cudaStream_t stream) {
  if (!X || !stage_group || !Y || nW < 0 || S < 1 || S > 32 || K < 1 || K > 32 || nW > (int64_t(1) << 40))
    return SF_EINVAL;
  for (int64_t s = 0; s < S; ++s)
    if (stage_group[s] < 0 || stage_group[s] >= K) return SF_EINVAL;
  if (!aligned(X, 8) || !aligned(Y, 8)) return SF_EINVAL_ALIGN;
  if (nW == 0) return SF_OK;
  return cuda_status(launch_stage_group_sum(X, nW, S, stage_group, K, Y, stream));
}

sf_status sf_gathered_to_steps(const int64_t* src, int64_t T, int64_t R, int64_t S, int64_t N, int64_t* dst,
                               cudaStream_t stream) {
  if (!src || !dst || !shape_ok(T, R, S) || N < 1) return SF_EINVAL;
  const uintptr_t a = reinterpret_cast<uintptr_t>(src), b = reinterpret_cast<uintptr_t>(dst);
  const uintptr_t bytes = uintptr_t(T) * uintptr_t(R) * uintptr_t(S) * 8u;
  if (a < b + bytes && b < a + bytes) return SF_EINVAL;  // the copy is not in place
  if (!aligned(src, 16) || !aligned(dst, 16)) return SF_EINVAL_ALIGN;
  return cuda_status(launch_gathered_to_steps(src, T, R, S, N, dst, stream));
}

sf_status sf_topk_suspects(const int64_t* X, const int64_t* E, int64_t nW, int64_t S, int64_t R, int32_t k,
                           int32_t* top_stage, int64_t* top_stage_value, int32_t* top_pair,
                           int64_t* top_pair_value, cudaStream_t stream) {
  if (!X || nW < 1 || nW > 0x7fffffff || S < 1 || S > 32 || R < 1 || R > 65536 || k < 1 || k > 32)
    return SF_EINVAL;
  if ((top_pair || top_pair_value) && !E) return SF_EINVAL;
  if (!top_stage && !top_stage_value && !top_pair && !top_pair_value) return SF_EINVAL;
  if (!aligned(X, 8) || !aligned(E, 8) || !aligned(top_stage, 4) || !aligned(top_stage_value, 8) ||
      !aligned(top_pair, 4) || !aligned(top_pair_value, 8))
    return SF_EINVAL_ALIGN;
  return cuda_status(
      launch_topk(X, E, nW, S, R, k, top_stage, top_stage_value, top_pair, top_pair_value, stream));
}

sf_status sf_window_median(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W, int64_t* m,
                           uint32_t* status, cudaStream_t stream) {
  // the median is defined for every int64 input; status only reports a bounded wait that ran out
  if (!d || !m || !shape_ok(T, R, S) || W < 1 || W > 65536) return SF_EINVAL;
  if (!aligned(d, 16) || !aligned(m, 8) || !aligned(status, 4)) return SF_EINVAL_ALIGN;
  const int64_t nW = (T + W - 1) / W;
  if (nW * ((R * S + 7) / 8) > 0x7fffffff) return SF_EUNSUPPORTED;
  return cuda_status(launch_window_median(d, T, R, S, W, m, status, stream));
}

sf_status sf_direct_gain(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W, const int64_t* m,
                         const int64_t* wall, int32_t other_stage, sf_ratio eta_Q, int64_t* X, int64_t* Y,
                         int64_t* D, int64_t* E, int32_t* C, uint8_t* step_lead, uint64_t* quality,
                         uint32_t* status, cudaStream_t stream) {
  if (!d || !m || !X || !Y || !D || !step_lead || !shape_ok(T, R, S) || W < 1 || W > 65536 ||
      other_stage < -1 || other_stage >= S || !ratio_ok(eta_Q))
    return SF_EINVAL;
  if (!aligned(d, 16) || !aligned(m, 8) || !aligned(wall, 8) || !aligned(X, 8) || !aligned(Y, 8) ||
      !aligned(D, 8) || !aligned(E, 8) || !aligned(C, 4) || !aligned(quality, 8) || !aligned(status, 4))
    return SF_EINVAL_ALIGN;
  const int64_t nW = (T + W - 1) / W;
  ZeroList z;
  z.add(X, size_t(nW) * S * 8);
  z.add(Y, size_t(nW) * S * 8);
  z.add(D, size_t(nW) * 8);
  z.add(E, size_t(nW) * S * R * 8);
  z.add(C, size_t(nW) * S * R * 4);
  z.add(quality, size_t(nW) * 6 * 8);
  bool cleared = false;
  cudaError_t e = launch_zero_many(z, stream, &cleared);
  if (e != cudaSuccess) return SF_ECUDA;
  StreamJob j;
  j.after_clear = cleared;
  j.d = d;
  j.T = T;
  j.R = R;
  j.S = S;
  j.X = X;
  j.D = D;
  j.E = E;
  j.C = C;
  j.step_lead = step_lead;
  j.W = W;
  j.gain = true;
  j.m = m;
  j.wall = wall;
  j.other_stage = other_stage;
  j.eta_num = eta_Q.num;
  j.eta_den = eta_Q.den;
  j.Y = Y;
  j.quality = (wall || other_stage >= 0) ? quality : nullptr;
  j.status = status;
  return cuda_status(launch_stream_pass(j, stream));
}

sf_status sf_label_gates(int64_t T, int64_t R, int64_t S, int64_t W, const int64_t* X, const int64_t* Y,
                         const int64_t* D, const uint8_t* step_lead, const uint64_t* quality,
                         const int32_t* role, const int32_t* missing, const sf_label_config* cfg,
                         uint32_t* labels, uint32_t* route_mask, uint32_t* amb_mask, double* share,
                         double* gain, int32_t* n_confident, int32_t* n_switch, cudaStream_t stream) {
  if (!X || !Y || !D || !step_lead || !labels || !route_mask || !amb_mask || !shape_ok(T, R, S) || W < 1 ||
      W > 65536 || !config_ok(cfg))
    return SF_EINVAL;
  if (!aligned(X, 8) || !aligned(Y, 8) || !aligned(D, 8) || !aligned(quality, 8) || !aligned(role, 4) ||
      !aligned(missing, 4) || !aligned(labels, 4) || !aligned(route_mask, 4) || !aligned(amb_mask, 4) ||
      !aligned(share, 8) || !aligned(gain, 8) || !aligned(n_confident, 4) || !aligned(n_switch, 4))
    return SF_EINVAL_ALIGN;
  GateJob g{};
  g.T = T;
  g.R = R;
  g.S = S;
  g.W = W;
  g.nW = (T + W - 1) / W;
  g.X = X;
  g.Y = Y;
  g.D = D;
  g.step_lead = step_lead;
  g.quality = quality;
  g.role = role;
  g.missing = missing;
  g.cfg = *cfg;
  g.labels = labels;
  g.route_mask = route_mask;
  g.amb_mask = amb_mask;
  g.share = share;
  g.gain = gain;
  g.n_confident = n_confident;
  g.n_switch = n_switch;
  return cuda_status(launch_gates(g, stream));
}

sf_status sf_selftest_bounded_wait(uint64_t limit_ns, uint32_t* status, cudaStream_t stream) {
  if (!status || limit_ns == 0 || limit_ns > kWaitLimitNs) return SF_EINVAL;
  if (!aligned(status, 4)) return SF_EINVAL_ALIGN;
  return cuda_status(launch_wait_selftest(limit_ns, status, stream));
}

size_t sf_label_windows_workspace_size(int64_t T, int64_t R, int64_t S, int64_t W) {
  if (!shape_ok(T, R, S) || W < 1 || W > 65536) return 0;
  return label_layout(T, R, S, W).total;
}

sf_status sf_label_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W, const int32_t* role,
                           const int32_t* missing, const int64_t* wall, int32_t other_stage,
                           const sf_label_config* cfg, void* workspace, size_t workspace_bytes,
                           uint32_t* labels, uint32_t* route_mask, uint32_t* amb_mask, double* share,
                           double* gain, int64_t* X, int64_t* Y, int64_t* D, uint32_t* status,
                           cudaStream_t stream) {
  if (!d || !labels || !route_mask || !amb_mask || !shape_ok(T, R, S) || W < 1 || W > 65536 ||
      other_stage < -1 || other_stage >= S || !config_ok(cfg))
    return SF_EINVAL;
  const LabelLayout L = label_layout(T, R, S, W);
  if (!workspace || workspace_bytes < L.total) return SF_EWORKSPACE;
  if (!aligned(workspace, 256) || !aligned(X, 8) || !aligned(Y, 8) || !aligned(D, 8)) return SF_EINVAL_ALIGN;
  unsigned char* ws = static_cast<unsigned char*>(workspace);
  int64_t* m = reinterpret_cast<int64_t*>(ws + L.m);
  int64_t* Xw = X ? X : reinterpret_cast<int64_t*>(ws + L.X);
  int64_t* Yw = Y ? Y : reinterpret_cast<int64_t*>(ws + L.Y);
  int64_t* Dw = D ? D : reinterpret_cast<int64_t*>(ws + L.D);
  uint64_t* q = reinterpret_cast<uint64_t*>(ws + L.q);
  uint8_t* sl = ws + L.sl;
  sf_status st = sf_window_median(d, T, R, S, W, m, status, stream);
  if (st != SF_OK) return st;
  st = sf_direct_gain(d, T, R, S, W, m, wall, other_stage, cfg->eta_Q, Xw, Yw, Dw, nullptr, nullptr, sl, q,
                      status, stream);
  if (st != SF_OK) return st;
  return sf_label_gates(T, R, S, W, Xw, Yw, Dw, sl, (wall || other_stage >= 0) ? q : nullptr, role, missing,
                        cfg, labels, route_mask, amb_mask, share, gain, nullptr, nullptr, stream);
}

}  // extern "C"

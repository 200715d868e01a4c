// The C ABI of libmilesloss: argument validation, workspace layout, launch
// planning and kernel launches. Nothing here allocates, frees or
// synchronises; every call enqueues its kernels on the caller's stream.
//
// rl_loss_fwd_bwd = advantage kernel -> fused sweep -> statistics kernel
// rl_loss_fwd     = advantage kernel -> forward-only sweep -> statistics kernel
// rl_loss_bwd     = gradient sweep from the saved per-row state
#include <climits>
#include <cmath>
#include <cstdlib>
#include <map>
#include <mutex>
#include <string>
#include <tuple>

#include "kernels.h"

using namespace milesloss;

namespace {
std::mutex g_ov_mu;
rl_launch_overrides g_ov = {-1, -1, -1, -1, -1, -1, -1, -1, -1, -1, -1, -1, -1};
}  // namespace

namespace milesloss {
rl_launch_overrides current_overrides() {
  std::lock_guard<std::mutex> lk(g_ov_mu);
  return g_ov;
}

rl_status status_of_bits(uint32_t bits) {
  for (int code = RL_ERR_TARGET_OUT_OF_RANGE; code <= RL_ERR_TOPK_ID_OUT_OF_RANGE; ++code)
    if (bits & (1u << code)) return static_cast<rl_status>(code);
  return RL_OK;
}
}  // namespace milesloss

namespace {

thread_local cudaEvent_t t_ev_begin = nullptr;
thread_local cudaEvent_t t_ev_end = nullptr;

std::mutex g_mu;
std::map<std::pair<int, const void*>, int> g_smem_set;               // (device, fn) -> bytes
std::map<std::tuple<int, const void*, int, int>, int> g_occupancy;   // (dev, fn, C, smem) -> clusters

bool finite(float x) { return std::isfinite(x); }

rl_status cuda_fail(cudaError_t e) { return e == cudaSuccess ? RL_OK : RL_ERR_CUDA; }

rl_status set_smem(const void* fn, int dev, int bytes) {
  std::lock_guard<std::mutex> lk(g_mu);
  auto key = std::make_pair(dev, fn);
  auto it = g_smem_set.find(key);
  if (it != g_smem_set.end() && it->second >= bytes) return RL_OK;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return RL_ERR_CUDA;
  g_smem_set[key] = bytes;
  return RL_OK;
}

// Number of clusters of C CTAs that can be resident at once.
rl_status resident_clusters(const void* fn, int dev, int C, int smem, int threads, int* out) {
  {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_occupancy.find(std::make_tuple(dev, fn, C, smem));
    if (it != g_occupancy.end()) { *out = it->second; return RL_OK; }
  }
  int n = 0;
  if (C == 1) {
    int per_sm = 0, sms = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, threads, smem) != cudaSuccess)
      return RL_ERR_CUDA;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return RL_ERR_CUDA;
    n = per_sm * sms;
  } else {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(C);
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = C;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) return RL_ERR_CUDA;
  }
  if (n <= 0) return RL_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lk(g_mu);
  g_occupancy[std::make_tuple(dev, fn, C, smem)] = n;
  *out = n;
  return RL_OK;
}

rl_status launch(const void* fn, dim3 grid, dim3 block, int smem, int cluster, cudaStream_t s,
                 void* arg) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  if (cluster > 1) {
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = cluster;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
  }
  void* args[1] = {arg};
  return cuda_fail(cudaLaunchKernelExC(&cfg, fn, args));
}

size_t elem_size(rl_dtype d) { return d == RL_BF16 ? 2 : 4; }
bool dtype_ok(int d) { return d == RL_BF16 || d == RL_F32; }
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

rl_status check_params(const rl_loss_params* p) {
  if (!p) return RL_ERR_INVALID_ARG;
  if (!finite(p->temperature) || !(p->temperature > 0.0f)) return RL_ERR_INVALID_ARG;
  if (!finite(p->eps_lo) || !finite(p->eps_hi) || p->eps_lo < 0.0f || p->eps_hi < 0.0f)
    return RL_ERR_INVALID_ARG;
  if (!finite(p->dual_clip_c) || p->dual_clip_c < 0.0f ||
      (p->dual_clip_c > 0.0f && p->dual_clip_c <= 1.0f))
    return RL_ERR_INVALID_ARG;
  if (!finite(p->kl_coef) || p->kl_coef < 0.0f) return RL_ERR_INVALID_ARG;
  if (!finite(p->entropy_coef) || p->entropy_coef < 0.0f) return RL_ERR_INVALID_ARG;
  if (!finite(p->std_floor) || !(p->std_floor > 0.0f)) return RL_ERR_INVALID_ARG;
  if ((p->normalize_std != 0 && p->normalize_std != 1) ||
      (p->unbiased_std != 0 && p->unbiased_std != 1))
    return RL_ERR_INVALID_ARG;
  if (p->correction < RL_CORR_NONE || p->correction > RL_CORR_CLIP_OR_POP)
    return RL_ERR_INVALID_ARG;
  if (p->correction != RL_CORR_NONE &&
      (!finite(p->corr_lo) || !finite(p->corr_hi) || p->corr_lo < 0.0f || p->corr_lo > p->corr_hi))
    return RL_ERR_INVALID_ARG;
  if (!finite(p->opd_coef)) return RL_ERR_INVALID_ARG;
  if (p->estimator < RL_EST_GRPO || p->estimator > RL_EST_GSPO) return RL_ERR_INVALID_ARG;
  if (p->opd_topk < 0 || p->opd_topk > kMaxTopK) return RL_ERR_INVALID_ARG;
  return RL_OK;
}

LossScalars scalars(const rl_loss_params* p) {
  LossScalars s;
  s.invT = 1.0f / p->temperature;
  s.k = 1.4426950408889634f / p->temperature;
  s.eps_lo = p->eps_lo;
  s.eps_hi = p->eps_hi;
  s.dual_c = p->dual_clip_c;
  s.beta = p->kl_coef;
  s.gamma = p->entropy_coef;
  s.corr_lo = p->corr_lo;
  s.corr_hi = p->corr_hi;
  s.corr = p->correction;
  const bool topk = p->opd_topk > 0 && p->opd_coef != 0.0f;
  s.topk = topk ? p->opd_topk : 0;
  s.opd_coef = p->opd_coef;
  s.topk_ids = topk ? p->opd_topk_ids : nullptr;
  s.topk_teacher = topk ? p->opd_topk_teacher : nullptr;
  return s;
}

struct SweepPlan {
  int C, S, slice, stage_bytes, smem, threads, variant;
};

// Several CTAs per SM hide each other's per-row synchronisation, so the
// plan aims at five CTAs of 256 threads per SM: the smallest cluster whose
// per-CTA slice fits a fifth of the SM's shared memory, then as many ring
// stages as still fit; if no cluster size fits, one CTA per SM.
// rl_set_launch_overrides can force the cluster size, stages and block shape.
constexpr long long kMinSliceBytes = 32 * 1024;  // smallest cluster slice a fused plan takes

rl_status plan_sweep(rl_dtype dt, long long V, int dev, int extra, bool grad,
                     const rl_launch_overrides& ov, SweepPlan* out) {
  int optin = 0, per_sm = 0, reserved = 0;
  if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev) !=
          cudaSuccess)
    return RL_ERR_CUDA;
  // Block shapes compiled: 256 threads for 5 or 4 CTAs per SM (48 or 64
  // registers), 512 threads for 2 CTAs per SM.
  const int threads = ov.cluster_threads > 0 ? ov.cluster_threads : 256;
  const int target = ov.cluster_ctas_per_sm > 0 ? ov.cluster_ctas_per_sm : (threads == 256 ? 5 : 2);
  if (!((threads == 256 && (target == 4 || target == 5)) || (threads == 512 && target == 2)))
    return RL_ERR_UNSUPPORTED;
  const int variant = threads == 512 ? 512 : (target == 5 ? 255 : 256);
  const int es = static_cast<int>(elem_size(dt));
  const int vec = 16 / es;
  const int forced_c = ov.cluster_size > 0 ? ov.cluster_size : 0;
  const int forced_s = ov.cluster_stages > 0 ? ov.cluster_stages : 0;
  const int fixed = kSweepSmemExtra + extra;                           // scratch (+ top-K)
  const int hard = optin - fixed;                                      // one CTA per SM
  const int share = per_sm / target - reserved - fixed;                // `target` per SM
  auto slice_of = [&](int C) {
    long long slice = (V + C - 1) / C;
    return (slice + vec - 1) / vec * vec;
  };
  auto fill = [&](int C, int S) {
    const long long slice = slice_of(C);
    const long long stage = (slice * es + 127) / 128 * 128;
    out->C = C;
    out->S = S;
    out->slice = static_cast<int>(slice);
    out->stage_bytes = static_cast<int>(stage);
    out->smem = static_cast<int>(S * stage) + fixed;
    out->threads = threads;
    out->variant = variant;
  };
  // Forward-only calls: one stage of the smallest slice that fits about a
  // third of the SM's shared memory, so three CTAs share an SM with bigger,
  // fewer copies and exchanges per row than in the fused call's plan. Measured
  // on GB300 against the fused plan: fp32 rows of 32,768 columns 2.36 against
  // 2.73 ms; bf16 rows of 32,768 and 65,536 columns 17-18 % faster. (Fused
  // calls keep the plan below: two stages of such slices were faster only for
  // fp32, by 1 %, and up to 24 % slower for bf16 rows.)
  if (!grad && !forced_c && !forced_s && threads == 256 && target == 5) {
    const int third = per_sm / 3 - reserved - fixed;
    const int S = 1;
    for (int C = 1; C <= kMaxCluster; C *= 2) {
      const long long slice = slice_of(C);
      if (C > 1 && slice * (C - 1) >= V) continue;
      const long long stage = (slice * es + 127) / 128 * 128;
      if (S * stage <= third) {
        fill(C, S);
        return RL_OK;
      }
    }
  }
  // Fused calls: for bf16 rows, the cluster of 2 or more CTAs whose slices
  // are 48-64 KB when there is one; otherwise (and for fp32) the largest cluster whose slices
  // are still at least kMinSliceBytes; as many stages as fit a fifth of the
  // SM's shared memory, else one. Measured on GB300 (bf16 rows): 20-24 KB
  // slices ran 10-25 % slower than 32-64 KB ones (40,960 / 49,152 columns),
  // 64 KB slices beat 32 KB ones by 2-7 % (65,536 / 131,072 columns); for
  // fp32 rows of 32,768 columns 32 KB slices beat 64 KB ones by 3 %.
  if (grad && !forced_c && !forced_s && threads == 256 && target == 5) {
    int C = 1;
    for (int c = 2; c <= kMaxCluster; c *= 2) {
      const long long slice = slice_of(c);
      if (slice * (c - 1) >= V || slice * es < kMinSliceBytes) break;
      C = c;
    }
    if (dt == RL_BF16) {
      for (int c = 2; c <= kMaxCluster; c *= 2) {  // (a whole 64 KB row in one CTA was slower)
        const long long b = slice_of(c) * es;
        if (b >= 48 * 1024 && b <= 64 * 1024 && slice_of(c) * (c - 1) < V) {
          C = c;
          break;
        }
      }
    }
    const long long stage = (slice_of(C) * es + 127) / 128 * 128;
    if (stage <= hard) {
      int S = stage <= share ? static_cast<int>(share / stage) : 1;
      if (S > kMaxStages) S = kMaxStages;
      fill(C, S);
      return RL_OK;
    }
  }
  for (int pass = 0; pass < 2; ++pass) {
    const int budget = pass == 0 ? share : hard;
    for (int C = 1; C <= kMaxCluster; C *= 2) {
      if (forced_c && C != forced_c) continue;
      long long slice = (V + C - 1) / C;
      slice = (slice + vec - 1) / vec * vec;
      if (C > 1 && slice * (C - 1) >= V) continue;  // every CTA must own columns
      const long long stage = (slice * es + 127) / 128 * 128;
      if (stage > budget) continue;
      int S = static_cast<int>(budget / stage);
      if (S > kMaxStages) S = kMaxStages;
      if (forced_s) {
        if (forced_s < 1 || forced_s > kMaxStages || forced_s * stage > hard)
          return RL_ERR_UNSUPPORTED;
        S = forced_s;
      }
      out->C = C;
      out->S = S;
      out->slice = static_cast<int>(slice);
      out->stage_bytes = static_cast<int>(stage);
      out->smem = static_cast<int>(S * stage) + fixed;
      out->threads = threads;
      out->variant = variant;
      return RL_OK;
    }
  }
  return RL_ERR_UNSUPPORTED;  // vocabulary too large for an 8-CTA cluster
}

struct Common {
  const void* logits;
  rl_dtype dt;
  long long R, V, ld;
  const int32_t* targets;
  const uint8_t* mask;
  const rl_loss_params* p;
};

rl_status check_common(const Common& c, bool need_logits = true) {
  if (!dtype_ok(c.dt)) return RL_ERR_INVALID_ARG;
  if (c.R < 0 || c.V < 1 || c.V > INT_MAX / 8 || c.ld < c.V) return RL_ERR_INVALID_ARG;
  if (c.R > 0 && ((need_logits && !c.logits) || !c.targets || !c.mask)) return RL_ERR_INVALID_ARG;
  return check_params(c.p);
}

struct FwdIn {
  Common c;
  const float *rho, *q, *old, *teacher, *rewards;
  const int32_t *gid, *cu;
  int n_traj, n_groups;
  float *out_logp, *out_H, *out_adv;
  int32_t* out_gsize;
  rl_loss_stats* stats;
  void* ws;
  size_t ws_bytes;
  // a shard of a row-sharded call (rl_loss_shard_fwd_bwd)
  long long row0 = 0;           // global index of the shard's first row
  long long R_total = -1;       // rows of the whole call (-1: c.R)
  const int* counts_in = nullptr;
  int* counts_out = nullptr;
  rl_loss_partials* part_out = nullptr;
  // a column shard of a vocabulary-sharded call (rl_loss_vocab_shard_fwd_bwd):
  // the logits are columns [col0, col0 + V); part_rows receives each row's
  // partial sums in place of the sweep's epilogue
  long long col0 = 0;
  int vocab_total = 0;  // the vocabulary's size (0: V)
  float4* part_rows = nullptr;
  // a shard of a sharded GSPO call: the per-trajectory sums over its rows go
  // here (k_seq's first half) and the call stops before the statistics
  double* seq_sums_out = nullptr;
};

rl_status check_fwd(const FwdIn& f, bool need_logits = true) {
  rl_status st = check_common(f.c, need_logits);
  if (st != RL_OK) return st;
  const rl_loss_params* p = f.c.p;
  if (f.n_traj < 0 || f.n_groups < 0) return RL_ERR_INVALID_ARG;
  if (f.n_traj > 0 && (f.n_groups < 1 || !f.rewards || !f.gid)) return RL_ERR_INVALID_ARG;
  if (!f.cu) return RL_ERR_INVALID_ARG;
  if (f.c.R > 0 && !f.rho) return RL_ERR_INVALID_ARG;
  if (f.c.R > 0 && p->kl_coef > 0.0f && !f.q) return RL_ERR_INVALID_ARG;
  if (f.c.R > 0 && p->opd_coef != 0.0f && p->opd_topk == 0 && !f.teacher)
    return RL_ERR_INVALID_ARG;
  if (f.c.R > 0 && p->opd_coef != 0.0f && p->opd_topk > 0 &&
      (!p->opd_topk_ids || !p->opd_topk_teacher ||
       (reinterpret_cast<uintptr_t>(p->opd_topk_ids) & 3u) ||
       (reinterpret_cast<uintptr_t>(p->opd_topk_teacher) & 3u)))
    return RL_ERR_INVALID_ARG;
  // GSPO scores whole trajectories with one advantage: no per-token shaping
  if (p->estimator == RL_EST_GSPO && p->opd_coef != 0.0f) return RL_ERR_UNSUPPORTED;
  if (!f.ws || (reinterpret_cast<uintptr_t>(f.ws) & 255u)) return RL_ERR_INVALID_ARG;
  size_t need = 0;
  rl_loss_workspace_size(f.c.R, f.n_traj, f.n_groups, &need);
  if (f.ws_bytes < need) return RL_ERR_WORKSPACE_TOO_SMALL;
  return RL_OK;
}

struct GradOut {
  float g;
  const float* g_dev;
  void* dl;
  rl_dtype dt;
  long long ld_out;
};

rl_status check_grad(const Common& c, const GradOut& o, bool need_out = true) {
  if (!finite(o.g)) return RL_ERR_INVALID_ARG;
  if (!dtype_ok(o.dt)) return RL_ERR_INVALID_ARG;
  if (o.ld_out < c.V) return RL_ERR_INVALID_ARG;
  if (c.R > 0 && need_out && !o.dl) return RL_ERR_INVALID_ARG;
  return RL_OK;
}

// The per-row arrays of a workspace view shifted to start at row r0.
WsPtrs rows_from(WsPtrs w, long long r0) {
  w.a_row += r0;
  w.logp += r0;
  w.H += r0;
  w.lse += r0;
  w.G += r0;
  w.ell += r0;
  w.pg += r0;
  w.k3 += r0;
  w.r += r0;
  w.rc += r0;
  w.flags += r0;
  return w;
}

template <class T>
T* shift(T* p, long long r0) { return p ? p + r0 : p; }

void record(cudaEvent_t ev, cudaStream_t s) {
  if (ev && t_ev_begin && t_ev_end) cudaEventRecord(ev, s);
}

// The gradient sweep from the per-row state in the workspace (lse, H, G).
rl_status launch_bwd(const Common& c, const GradOut& go, const WsPtrs& ws, cudaStream_t s,
                     long long col0 = 0) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return RL_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return RL_ERR_CUDA;
  BwdArgs b;
  b.logits = c.logits;
  b.ld = c.ld;
  b.R = c.R;
  b.V = static_cast<int>(c.V);
  b.tiles_per_row = static_cast<int>((c.V + kBwdTile - 1) / kBwdTile);
  b.n_tiles = c.R * b.tiles_per_row;
  b.in_vec = aligned16(c.logits) && ((c.ld * elem_size(c.dt)) % 16 == 0);
  b.out_vec = aligned16(go.dl) && ((go.ld_out * elem_size(go.dt)) % 16 == 0);
  b.targets = c.targets;
  b.mask = c.mask;
  b.dlogits = go.dl;
  b.ld_out = go.ld_out;
  b.grad_loss = go.g;
  b.grad_loss_dev = go.g_dev;
  b.invT = 1.0f / c.p->temperature;
  b.k = 1.4426950408889634f / c.p->temperature;
  b.gamma = c.p->entropy_coef;
  b.col0 = static_cast<int>(col0);  // vocabulary ids fit int32
  b.ws = ws;
  // one wave of resident blocks (grid-stride over the tiles): a second,
  // partial wave would run with fewer loads in flight
  const void* fn = bwd_kernel(c.dt, go.dt);
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kBwdThreads, 0) != cudaSuccess)
    return RL_ERR_CUDA;
  const long long grid =
      std::min<long long>(b.n_tiles, static_cast<long long>(sms) * std::max(per_sm, 1));
  return launch(fn, dim3(static_cast<unsigned>(grid)), dim3(kBwdThreads), 0, 1, s, &b);
}

// GSPO's per-trajectory pass over a call's rows (k_seq), whole or one half
// of a sharded call's (sums_out: the shard's sums only; sums_in: apply the
// sums added over the shards).
rl_status launch_seq(const FwdIn& f, double* sums_out, const double* sums_in, cudaStream_t s) {
  SeqArgs qa;
  qa.cu = f.cu;
  qa.rho = f.rho;
  qa.old = f.old;
  qa.q = f.q;
  qa.mask = f.c.mask;
  qa.row0 = f.row0;
  qa.R = f.c.R;
  qa.sums_out = sums_out;
  qa.sums_in = sums_in;
  qa.s = scalars(f.c.p);
  qa.ws = WsPtrs::at(f.ws, WsLayout::make(f.c.R, f.n_traj, f.n_groups));
  return launch(seq_kernel(), dim3(static_cast<unsigned>(f.n_traj)), dim3(kSeqThreads), 0, 1, s,
                &qa);
}

// A shard's partial statistics over its rows (k_stats into `partials`).
rl_status launch_shard_stats(const FwdIn& f, rl_loss_partials* partials, cudaStream_t s) {
  StatArgs ta;
  ta.R = f.c.R;
  ta.mask = f.c.mask;
  ta.rho = f.rho;
  ta.out = nullptr;
  ta.part_out = partials;
  ta.ws = WsPtrs::at(f.ws, WsLayout::make(f.c.R, f.n_traj, f.n_groups));
  long long blocks = (f.c.R + kStatThreads - 1) / kStatThreads;
  blocks = std::max<long long>(1, std::min<long long>(blocks, kMaxStatBlocks));
  return launch(stats_kernel(), dim3(static_cast<unsigned>(blocks)), dim3(kStatThreads), 0, 1, s,
                &ta);
}

// phase: RL_PHASE_BEGIN (advantages, N), RL_PHASE_ROWS (the sweep over rows
// [r0, r1), whose logits / dLogits pointers address row r0), RL_PHASE_END
// (the statistics); rl_loss_fwd / rl_loss_fwd_bwd run all three on [0, R).
rl_status run_fwd(const FwdIn& f, const GradOut* go, cudaStream_t s, int phase = RL_PHASE_ALL,
                  long long r0 = 0, long long r1 = -1) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return RL_ERR_CUDA;
  const Common& call = f.c;
  if (r1 < 0) r1 = call.R;
  const WsLayout L = WsLayout::make(call.R, f.n_traj, f.n_groups);
  const WsPtrs ws_all = WsPtrs::at(f.ws, L);
  rl_status st = RL_OK;

  if (phase & RL_PHASE_BEGIN) {
  const Common& c = call;
  const WsPtrs& ws = ws_all;
  // advantages, N, validation
  AdvArgs aa;
  aa.R = c.R;
  aa.row0 = f.row0;
  aa.R_total = f.R_total >= 0 ? f.R_total : c.R;
  aa.counts_in = f.counts_in;
  aa.counts_out = f.counts_out;
  aa.n_traj = f.n_traj;
  aa.n_groups = f.n_groups;
  aa.rewards = f.rewards;
  aa.gid = f.gid;
  aa.cu = f.cu;
  aa.mask = c.mask;
  aa.rho = f.rho;
  aa.teacher = (c.p->opd_coef != 0.0f && c.p->opd_topk == 0) ? f.teacher : nullptr;
  aa.opd_coef = c.p->opd_coef;
  aa.normalize_std = c.p->normalize_std;
  aa.unbiased_std = c.p->unbiased_std;
  aa.std_floor = c.p->std_floor;
  aa.advantages = f.out_adv;
  aa.group_sizes = f.out_gsize;
  aa.estimator = c.p->estimator;
  // cu_seqlens, per-trajectory counts and advantages, group ids, rewards
  const size_t traj_bytes = (5 * static_cast<size_t>(f.n_traj) + 1) * sizeof(int);
  aa.smem_traj = traj_bytes <= static_cast<size_t>(kAdvSmemBytes);
  aa.ws = ws;
  if (f.n_groups > kInlineGroups) {
    const int gb = std::min(f.n_groups, kMaxGroupBlocks);
    st = launch(groups_kernel(), dim3(static_cast<unsigned>(gb)), dim3(32), 0, 1, s, &aa);
    if (st != RL_OK) return st;
  }
  st = launch(adv_kernel(), dim3(1), dim3(kAdvThreads),
              aa.smem_traj ? static_cast<int>(traj_bytes) : 0, 1, s, &aa);
  if (st != RL_OK) return st;
  }

  // GSPO: the gradient of a token depends on its whole trajectory, so the
  // call runs as forward sweep -> per-trajectory pass -> gradient sweep.
  const bool gspo = call.p->estimator == RL_EST_GSPO;
  const GradOut* go_sweep = gspo ? nullptr : go;

  // the sweep sees rows [r0, r1) as a call of its own: per-row pointers and
  // the workspace's per-row arrays start at row r0
  Common c = call;
  c.R = (phase & RL_PHASE_ROWS) ? r1 - r0 : 0;
  c.targets = shift(call.targets, r0);
  c.mask = shift(call.mask, r0);
  FwdIn fr = f;
  fr.c = c;
  fr.rho = shift(f.rho, r0);
  fr.q = shift(f.q, r0);
  fr.old = shift(f.old, r0);
  fr.out_logp = shift(f.out_logp, r0);
  fr.out_H = shift(f.out_H, r0);
  const WsPtrs ws = rows_from(ws_all, r0);
  LossScalars sc = scalars(call.p);
  if (sc.topk) {
    sc.topk_ids = shift(sc.topk_ids, r0 * sc.topk);
    sc.topk_teacher = shift(sc.topk_teacher, r0 * sc.topk);
  }

  const bool grad = go_sweep != nullptr;
  const size_t es = elem_size(c.dt);
  const bool in_bulk = aligned16(c.logits) && ((c.ld * es) % 16 == 0);
  const bool out_vec = grad && aligned16(go->dl) && ((go->ld_out * elem_size(go->dt)) % 16 == 0);
  const rl_launch_overrides ov = current_overrides();
  const unsigned long long stall =
      ov.stall_first_wait_ns > 0 ? static_cast<unsigned long long>(ov.stall_first_wait_ns) : 0ull;
  if (c.R > 0 &&
      use_stream(c.V * static_cast<long long>(es), static_cast<int>(es), in_bulk, grad, sc.topk > 0, ov)) {
    StreamPlan sp;
    const void* fn = nullptr;
    int ctas = 0;  // resident CTAs, or clusters of sp.cluster CTAs
    int threads = 0;
    rl_launch_overrides pov = ov;
    for (;;) {
      st = plan_stream(dev, sc.topk ? kTopKSmem : 0, c.V * static_cast<long long>(es),
                       static_cast<int>(es), grad, sc.topk > 0, f.part_rows == nullptr, pov, &sp);
      if (st != RL_OK) return st;
      fn = stream_kernel(c.dt, grad ? go->dt : c.dt, grad, sc.topk > 0, sp.cw, sp.cluster > 1);
      if (!fn) return RL_ERR_UNSUPPORTED;
      st = set_smem(fn, dev, sp.smem);
      if (st != RL_OK) return st;
      threads = stream_threads(sc.topk > 0, sp.cw);
      st = resident_clusters(fn, dev, sp.cluster, sp.smem, threads, &ctas);
      // no cluster of the plan fits the device (a partition with too few SMs
      // together): one CTA per row instead, unless the override forced it
      if (st == RL_ERR_UNSUPPORTED && sp.cluster > 1 && ov.stream_cluster <= 0) {
        pov.stream_cluster = 1;
        continue;
      }
      if (st != RL_OK) return st;
      break;
    }
    StreamArgs ta;
    ta.logits = c.logits;
    ta.ld = c.ld;
    ta.R = c.R;
    ta.V = static_cast<int>(c.V);
    ta.chunk_bytes = sp.chunk;
    ta.n_slots = sp.slots;
    ta.n_hold = sp.hold;
    ta.split_first = sp.split_first;
    ta.prefetch = sp.prefetch;
    ta.out_vec = out_vec;
    ta.slice_vec = sp.slice_vec;
    ta.targets = c.targets;
    ta.rho = fr.rho;
    ta.q = fr.q;
    ta.old = fr.old;
    ta.mask = c.mask;
    ta.out_logp = fr.out_logp;
    ta.out_H = fr.out_H;
    ta.dlogits = grad ? go->dl : nullptr;
    ta.ld_out = grad ? go->ld_out : 0;
    ta.grad_loss = grad ? go->g : 0.0f;
    ta.grad_loss_dev = grad ? go->g_dev : nullptr;
    ta.s = sc;
    ta.ws = ws;
    ta.stall_ns = stall;
    ta.col0 = f.col0;
    ta.vocab_total = f.vocab_total > 0 ? f.vocab_total : ta.V;
    ta.part_rows = shift(f.part_rows, 2 * r0);
    const long long grid = std::min<long long>(ctas, c.R) * sp.cluster;
    record(t_ev_begin, s);
    st = launch(fn, dim3(static_cast<unsigned>(grid)), dim3(threads), sp.smem, sp.cluster, s,
                &ta);
    record(t_ev_end, s);
    if (st != RL_OK) return st;
  } else if (c.R > 0) {
    SweepPlan pl;
    st = plan_sweep(c.dt, c.V, dev, sc.topk ? kTopKSmem : 0, grad, ov, &pl);
    if (st != RL_OK) return st;
    const void* fn = sweep_kernel(c.dt, grad ? go->dt : c.dt, grad, pl.variant, sc.topk > 0);
    st = set_smem(fn, dev, pl.smem);
    if (st != RL_OK) return st;
    int clusters = 0;
    st = resident_clusters(fn, dev, pl.C, pl.smem, pl.threads, &clusters);
    if (st != RL_OK) return st;
    const long long n_cl = std::min<long long>(clusters, c.R);

    SweepArgs sa;
    sa.logits = c.logits;
    sa.ld = c.ld;
    sa.R = c.R;
    sa.V = static_cast<int>(c.V);
    sa.slice = pl.slice;
    sa.stages = pl.S;
    sa.stage_bytes = pl.stage_bytes;
    sa.in_bulk = in_bulk;
    sa.out_vec = out_vec;
    sa.targets = c.targets;
    sa.rho = fr.rho;
    sa.q = fr.q;
    sa.old = fr.old;
    sa.mask = c.mask;
    sa.out_logp = fr.out_logp;
    sa.out_H = fr.out_H;
    sa.dlogits = grad ? go->dl : nullptr;
    sa.ld_out = grad ? go->ld_out : 0;
    sa.grad_loss = grad ? go->g : 0.0f;
    sa.grad_loss_dev = grad ? go->g_dev : nullptr;
    sa.s = sc;
    sa.ws = ws;
    sa.stall_ns = stall;
    sa.col0 = f.col0;
    sa.vocab_total = f.vocab_total > 0 ? f.vocab_total : sa.V;
    sa.part_rows = shift(f.part_rows, 2 * r0);
    record(t_ev_begin, s);
    st = launch(fn, dim3(static_cast<unsigned>(n_cl * pl.C)), dim3(pl.threads), pl.smem, pl.C,
                s, &sa);
    record(t_ev_end, s);
    if (st != RL_OK) return st;
  }

  if (gspo && (phase & RL_PHASE_ROWS) && (call.R > 0 || f.seq_sums_out) && f.n_traj > 0) {
    st = launch_seq(f, f.seq_sums_out, nullptr, s);
    if (st != RL_OK) return st;
  }

  if ((phase & RL_PHASE_END) && (f.stats || f.part_out)) {
    StatArgs ta;
    ta.R = call.R;
    ta.mask = call.mask;
    ta.rho = f.rho;
    ta.out = f.stats;
    ta.part_out = f.part_out;
    ta.ws = ws_all;
    long long blocks = (call.R + kStatThreads - 1) / kStatThreads;  // one row per thread
    blocks = std::max<long long>(1, std::min<long long>(blocks, kMaxStatBlocks));
    st = launch(stats_kernel(), dim3(static_cast<unsigned>(blocks)), dim3(kStatThreads), 0, 1, s,
                &ta);
    if (st != RL_OK) return st;
  }
  if (gspo && go && (phase & RL_PHASE_ROWS) && call.R > 0) return launch_bwd(call, *go, ws_all, s);
  return RL_OK;
}

}  // namespace

extern "C" {

rl_status rl_loss_workspace_size(int64_t n_rows, int32_t n_traj, int32_t n_groups, size_t* bytes) {
  if (!bytes || n_rows < 0 || n_traj < 0 || n_groups < 0) return RL_ERR_INVALID_ARG;
  *bytes = WsLayout::make(n_rows, n_traj, n_groups).total;
  return RL_OK;
}

rl_status rl_loss_fwd(const void* logits, rl_dtype logits_dtype, int64_t n_rows, int64_t vocab,
                      int64_t ld, const int32_t* targets, const float* rollout_logprobs,
                      const float* ref_logprobs, const float* old_logprobs,
                      const float* teacher_logprobs, const float* rewards,
                      const int32_t* group_id, const int32_t* cu_seqlens, int32_t n_traj,
                      int32_t n_groups, const uint8_t* loss_mask, const rl_loss_params* params,
                      float* token_logprobs, float* entropy, float* advantages,
                      int32_t* group_sizes, rl_loss_stats* stats, void* workspace,
                      size_t workspace_bytes, rl_stream stream) {
  FwdIn f{{logits, logits_dtype, n_rows, vocab, ld, targets, loss_mask, params},
          rollout_logprobs, ref_logprobs, old_logprobs, teacher_logprobs, rewards,
          group_id, cu_seqlens, n_traj, n_groups, token_logprobs, entropy, advantages,
          group_sizes, stats, workspace, workspace_bytes};
  rl_status st = check_fwd(f);
  if (st != RL_OK) return st;
  return run_fwd(f, nullptr, reinterpret_cast<cudaStream_t>(stream));
}

rl_status rl_loss_fwd_bwd(const void* logits, rl_dtype logits_dtype, int64_t n_rows,
                          int64_t vocab, int64_t ld, const int32_t* targets,
                          const float* rollout_logprobs, const float* ref_logprobs,
                          const float* old_logprobs, const float* teacher_logprobs,
                          const float* rewards, const int32_t* group_id,
                          const int32_t* cu_seqlens, int32_t n_traj, int32_t n_groups,
                          const uint8_t* loss_mask, const rl_loss_params* params,
                          float* token_logprobs, float* entropy, float* advantages,
                          int32_t* group_sizes, rl_loss_stats* stats, float grad_loss,
                          const float* grad_loss_device, void* dlogits, rl_dtype dlogits_dtype,
                          int64_t ld_out, void* workspace, size_t workspace_bytes,
                          rl_stream stream) {
  FwdIn f{{logits, logits_dtype, n_rows, vocab, ld, targets, loss_mask, params},
          rollout_logprobs, ref_logprobs, old_logprobs, teacher_logprobs, rewards,
          group_id, cu_seqlens, n_traj, n_groups, token_logprobs, entropy, advantages,
          group_sizes, stats, workspace, workspace_bytes};
  rl_status st = check_fwd(f);
  if (st != RL_OK) return st;
  GradOut go{grad_loss, grad_loss_device, dlogits, dlogits_dtype, ld_out};
  st = check_grad(f.c, go);
  if (st != RL_OK) return st;
  return run_fwd(f, &go, reinterpret_cast<cudaStream_t>(stream));
}

rl_status rl_loss_fwd_bwd_rows(int32_t phase, int64_t row_begin, int64_t row_end,
                               const void* logits, rl_dtype logits_dtype, int64_t n_rows,
                               int64_t vocab, int64_t ld, const int32_t* targets,
                               const float* rollout_logprobs, const float* ref_logprobs,
                               const float* old_logprobs, const float* teacher_logprobs,
                               const float* rewards, const int32_t* group_id,
                               const int32_t* cu_seqlens, int32_t n_traj, int32_t n_groups,
                               const uint8_t* loss_mask, const rl_loss_params* params,
                               float* token_logprobs, float* entropy, float* advantages,
                               int32_t* group_sizes, rl_loss_stats* stats, float grad_loss,
                               const float* grad_loss_device, void* dlogits,
                               rl_dtype dlogits_dtype, int64_t ld_out, void* workspace,
                               size_t workspace_bytes, rl_stream stream) {
  if (phase < 1 || phase > RL_PHASE_ALL) return RL_ERR_INVALID_ARG;
  if (row_begin < 0 || row_end < row_begin || row_end > n_rows) return RL_ERR_INVALID_ARG;
  const bool sweep = (phase & RL_PHASE_ROWS) && row_end > row_begin;
  FwdIn f{{logits, logits_dtype, n_rows, vocab, ld, targets, loss_mask, params},
          rollout_logprobs, ref_logprobs, old_logprobs, teacher_logprobs, rewards,
          group_id, cu_seqlens, n_traj, n_groups, token_logprobs, entropy, advantages,
          group_sizes, stats, workspace, workspace_bytes};
  rl_status st = check_fwd(f, sweep);
  if (st != RL_OK) return st;
  GradOut go{grad_loss, grad_loss_device, dlogits, dlogits_dtype, ld_out};
  const bool grad = dlogits != nullptr;  // NULL: the chunk runs forward-only
  if (grad) {
    st = check_grad(f.c, go, sweep);
    if (st != RL_OK) return st;
  }
  // GSPO needs every row's log-prob before any gradient: whole calls only
  if (params->estimator == RL_EST_GSPO && (phase != RL_PHASE_ALL || row_begin != 0 ||
                                           row_end != n_rows))
    return RL_ERR_UNSUPPORTED;
  return run_fwd(f, grad ? &go : nullptr, reinterpret_cast<cudaStream_t>(stream), phase,
                 row_begin, row_end);
}

rl_status rl_loss_shard_fwd_bwd(int32_t phase, int64_t row_offset, int64_t n_rows_total,
                                const void* logits, rl_dtype logits_dtype, int64_t n_rows,
                                int64_t vocab, int64_t ld, const int32_t* targets,
                                const float* rollout_logprobs, const float* ref_logprobs,
                                const float* old_logprobs, const float* teacher_logprobs,
                                const float* rewards, const int32_t* group_id,
                                const int32_t* cu_seqlens, int32_t n_traj, int32_t n_groups,
                                const uint8_t* loss_mask, const rl_loss_params* params,
                                float* token_logprobs, float* entropy, float* advantages,
                                int32_t* group_sizes, int32_t* traj_counts, double* traj_sums,
                                rl_loss_partials* partials, rl_loss_stats* stats,
                                float grad_loss, const float* grad_loss_device, void* dlogits,
                                rl_dtype dlogits_dtype, int64_t ld_out, void* workspace,
                                size_t workspace_bytes, rl_stream stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (phase == RL_SHARD_FINISH) {
    if (!partials || !stats) return RL_ERR_INVALID_ARG;
    FinishArgs fa{partials, stats};
    return launch(finish_kernel(), dim3(1), dim3(32), 0, 1, s, &fa);
  }
  if (phase != RL_SHARD_COUNT && phase != RL_SHARD_SWEEP && phase != RL_SHARD_SEQ)
    return RL_ERR_INVALID_ARG;
  if (row_offset < 0 || n_rows < 0 || n_rows_total < 0 || row_offset > n_rows_total - n_rows)
    return RL_ERR_INVALID_ARG;
  if (n_traj > 0 && !traj_counts) return RL_ERR_INVALID_ARG;
  if (!params) return RL_ERR_INVALID_ARG;
  // GSPO: a trajectory's sequence ratio needs its rows on every shard, so
  // its sweep stops at the per-trajectory sums, which the caller adds over
  // the shards before SEQ
  const bool gspo = params->estimator == RL_EST_GSPO;
  if (phase == RL_SHARD_SEQ && !gspo) return RL_ERR_INVALID_ARG;
  if (gspo && phase != RL_SHARD_COUNT && n_traj > 0 && !traj_sums) return RL_ERR_INVALID_ARG;
  const bool count = phase == RL_SHARD_COUNT;
  FwdIn f{{logits, logits_dtype, n_rows, vocab, ld, targets, loss_mask, params},
          rollout_logprobs, ref_logprobs, old_logprobs, teacher_logprobs, rewards,
          group_id, cu_seqlens, n_traj, n_groups, count ? nullptr : token_logprobs,
          count ? nullptr : entropy, count ? nullptr : advantages,
          count ? nullptr : group_sizes, nullptr, workspace, workspace_bytes};
  f.row0 = row_offset;
  f.R_total = n_rows_total;
  if (count) {
    f.counts_out = traj_counts;
    rl_status st = check_fwd(f, false);
    if (st != RL_OK) return st;
    return run_fwd(f, nullptr, s, RL_PHASE_BEGIN);
  }
  f.counts_in = traj_counts;
  if (phase == RL_SHARD_SWEEP && gspo) {
    // advantages, the forward sweep and the shard's per-trajectory sums
    f.seq_sums_out = traj_sums;
    rl_status st = check_fwd(f, n_rows > 0);
    if (st != RL_OK) return st;
    return run_fwd(f, nullptr, s, RL_PHASE_BEGIN | RL_PHASE_ROWS);
  }
  if (!partials) return RL_ERR_INVALID_ARG;
  GradOut go{grad_loss, grad_loss_device, dlogits, dlogits_dtype, ld_out};
  const bool grad = dlogits != nullptr;
  if (phase == RL_SHARD_SWEEP) {
    f.part_out = partials;
    rl_status st = check_fwd(f, n_rows > 0);
    if (st != RL_OK) return st;
    if (grad) {
      st = check_grad(f.c, go);
      if (st != RL_OK) return st;
    }
    return run_fwd(f, grad ? &go : nullptr, s, RL_PHASE_ALL);
  }
  // SEQ (GSPO): the trajectories' terms from the added sums, the shard's
  // partial statistics, dLogits over its rows
  rl_status st = check_fwd(f, n_rows > 0 && grad);
  if (st != RL_OK) return st;
  if (grad) {
    st = check_grad(f.c, go);
    if (st != RL_OK) return st;
  }
  if (n_traj > 0) {
    st = launch_seq(f, nullptr, traj_sums, s);
    if (st != RL_OK) return st;
  }
  st = launch_shard_stats(f, partials, s);
  if (st != RL_OK) return st;
  if (grad && n_rows > 0)
    return launch_bwd(f.c, go, WsPtrs::at(workspace, WsLayout::make(n_rows, n_traj, n_groups)), s);
  return RL_OK;
}

rl_status rl_loss_vocab_shard_fwd_bwd(
    int32_t phase, int32_t col_shard, int32_t n_col_shards, const int64_t* col_starts,
    int64_t row_offset, int64_t n_rows_total, const void* logits, rl_dtype logits_dtype,
    int64_t n_rows, int64_t ld, const int32_t* targets, const float* rollout_logprobs,
    const float* ref_logprobs, const float* old_logprobs, const float* teacher_logprobs,
    const float* rewards, const int32_t* group_id, const int32_t* cu_seqlens, int32_t n_traj,
    int32_t n_groups, const uint8_t* loss_mask, const rl_loss_params* params,
    float* token_logprobs, float* entropy, float* advantages, int32_t* group_sizes,
    int32_t* traj_counts, double* traj_sums, float* row_partials, const float* row_partials_all,
    rl_loss_partials* partials, rl_loss_stats* stats, float grad_loss,
    const float* grad_loss_device, void* dlogits, rl_dtype dlogits_dtype, int64_t ld_out,
    void* workspace, size_t workspace_bytes, rl_stream stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (phase == RL_VSHARD_FINISH) {
    if (!partials || !stats) return RL_ERR_INVALID_ARG;
    FinishArgs fa{partials, stats};
    return launch(finish_kernel(), dim3(1), dim3(32), 0, 1, s, &fa);
  }
  if (phase != RL_VSHARD_COUNT && phase != RL_VSHARD_PARTIAL && phase != RL_VSHARD_SWEEP &&
      phase != RL_VSHARD_SEQ)
    return RL_ERR_INVALID_ARG;
  // the column partition: col_starts[0] = 0 < col_starts[1] < ... (every
  // shard has a column), vocabulary ids fit the int32 targets
  if (n_col_shards < 1 || n_col_shards > kMaxColShards || !col_starts) return RL_ERR_INVALID_ARG;
  if (col_shard < 0 || col_shard >= n_col_shards || col_starts[0] != 0) return RL_ERR_INVALID_ARG;
  for (int k = 0; k < n_col_shards; ++k)
    if (col_starts[k + 1] <= col_starts[k]) return RL_ERR_INVALID_ARG;
  if (col_starts[n_col_shards] > INT32_MAX) return RL_ERR_INVALID_ARG;
  const long long col0 = col_starts[col_shard];
  const long long vocab = col_starts[col_shard + 1] - col0;
  if (row_offset < 0 || n_rows < 0 || n_rows_total < 0 || row_offset > n_rows_total - n_rows)
    return RL_ERR_INVALID_ARG;
  if (n_traj > 0 && !traj_counts) return RL_ERR_INVALID_ARG;
  if (!params) return RL_ERR_INVALID_ARG;
  // GSPO: SWEEP stops at the per-trajectory sums over the shard's rows, which
  // the caller adds over the row shards before SEQ
  const bool gspo = params->estimator == RL_EST_GSPO;
  if (phase == RL_VSHARD_SEQ && !gspo) return RL_ERR_INVALID_ARG;
  if (gspo && (phase == RL_VSHARD_SWEEP || phase == RL_VSHARD_SEQ) && n_traj > 0 && !traj_sums)
    return RL_ERR_INVALID_ARG;
  const bool count = phase == RL_VSHARD_COUNT;
  const bool sweep = phase == RL_VSHARD_SWEEP || phase == RL_VSHARD_SEQ;
  FwdIn f{{logits, logits_dtype, n_rows, vocab, ld, targets, loss_mask, params},
          rollout_logprobs, ref_logprobs, old_logprobs, teacher_logprobs, rewards,
          group_id, cu_seqlens, n_traj, n_groups, sweep ? token_logprobs : nullptr,
          sweep ? entropy : nullptr, count ? nullptr : advantages,
          count ? nullptr : group_sizes, nullptr, workspace, workspace_bytes};
  f.row0 = row_offset;
  f.R_total = n_rows_total;
  f.col0 = col0;
  f.vocab_total = static_cast<int>(col_starts[n_col_shards]);
  if (count) {
    f.counts_out = traj_counts;
    rl_status st = check_fwd(f, false);
    if (st != RL_OK) return st;
    return run_fwd(f, nullptr, s, RL_PHASE_BEGIN);
  }
  if (phase == RL_VSHARD_PARTIAL) {
    // advantages and N from the summed counts, then the forward sweep over
    // this shard's columns, writing each row's partial sums
    if (n_rows > 0 && (!row_partials || !aligned16(row_partials))) return RL_ERR_INVALID_ARG;
    f.counts_in = traj_counts;
    f.part_rows = reinterpret_cast<float4*>(row_partials);
    rl_status st = check_fwd(f, n_rows > 0);
    if (st != RL_OK) return st;
    return run_fwd(f, nullptr, s, RL_PHASE_BEGIN | RL_PHASE_ROWS);
  }
  // SWEEP: merge the gathered records, dLogits over this shard's columns,
  // this shard's partial statistics (GSPO: the merge and the shard's
  // per-trajectory sums; SEQ: the rest)
  if (!partials && !(gspo && phase == RL_VSHARD_SWEEP)) return RL_ERR_INVALID_ARG;
  if (phase == RL_VSHARD_SWEEP && n_rows > 0 &&
      (!row_partials_all || !aligned16(row_partials_all)))
    return RL_ERR_INVALID_ARG;
  GradOut go{grad_loss, grad_loss_device, dlogits, dlogits_dtype, ld_out};
  const bool grad = dlogits != nullptr && !(gspo && phase == RL_VSHARD_SWEEP);
  rl_status st = check_fwd(f, n_rows > 0 && grad);
  if (st != RL_OK) return st;
  if (grad) {
    st = check_grad(f.c, go);
    if (st != RL_OK) return st;
  }
  const WsPtrs ws = WsPtrs::at(workspace, WsLayout::make(n_rows, n_traj, n_groups));
  if (phase == RL_VSHARD_SEQ) {
    if (n_traj > 0) {
      st = launch_seq(f, nullptr, traj_sums, s);
      if (st != RL_OK) return st;
    }
    st = launch_shard_stats(f, partials, s);
    if (st != RL_OK) return st;
    if (grad && n_rows > 0) return launch_bwd(f.c, go, ws, s, col0);
    return RL_OK;
  }
  if (n_rows > 0) {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return RL_ERR_CUDA;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return RL_ERR_CUDA;
    MergeArgs ma;
    ma.R = n_rows;
    ma.n_shards = n_col_shards;
    for (int k = 0; k <= n_col_shards; ++k) ma.col_starts[k] = col_starts[k];
    ma.all = reinterpret_cast<const float4*>(row_partials_all);
    ma.targets = targets;
    ma.rho = rollout_logprobs;
    ma.q = ref_logprobs;
    ma.old = old_logprobs;
    ma.mask = loss_mask;
    ma.out_logp = token_logprobs;
    ma.out_H = entropy;
    ma.s = scalars(params);
    ma.ws = ws;
    const long long blocks = std::min<long long>((n_rows + kMergeThreads - 1) / kMergeThreads,
                                                 static_cast<long long>(sms) * 8);
    st = launch(merge_kernel(), dim3(static_cast<unsigned>(blocks)), dim3(kMergeThreads), 0, 1,
                s, &ma);
    if (st != RL_OK) return st;
  }
  if (gspo) return n_traj > 0 ? launch_seq(f, traj_sums, nullptr, s) : RL_OK;
  if (grad && n_rows > 0) {
    st = launch_bwd(f.c, go, ws, s, col0);
    if (st != RL_OK) return st;
  }
  return launch_shard_stats(f, partials, s);
}

rl_status rl_loss_bwd(const void* logits, rl_dtype logits_dtype, int64_t n_rows, int64_t vocab,
                      int64_t ld, const int32_t* targets, const uint8_t* loss_mask,
                      const rl_loss_params* params, float grad_loss,
                      const float* grad_loss_device, const void* workspace,
                      size_t workspace_bytes, void* dlogits, rl_dtype dlogits_dtype,
                      int64_t ld_out, rl_stream stream) {
  Common c{logits, logits_dtype, n_rows, vocab, ld, targets, loss_mask, params};
  rl_status st = check_common(c);
  if (st != RL_OK) return st;
  GradOut go{grad_loss, grad_loss_device, dlogits, dlogits_dtype, ld_out};
  st = check_grad(c, go);
  if (st != RL_OK) return st;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return RL_ERR_INVALID_ARG;
  const WsLayout L = WsLayout::make(n_rows, 0, 0);
  if (workspace_bytes < L.total) return RL_ERR_WORKSPACE_TOO_SMALL;
  if (n_rows == 0) return RL_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  record(t_ev_begin, s);
  st = launch_bwd(c, go, WsPtrs::at(const_cast<void*>(workspace), L), s);
  record(t_ev_end, s);
  return st;
}

rl_status rl_loss_check_device_error(const void* workspace) {
  if (!workspace) return RL_ERR_INVALID_ARG;
  uint32_t bits = 0;
  if (cudaMemcpy(&bits, workspace, sizeof(bits), cudaMemcpyDeviceToHost) != cudaSuccess)
    return RL_ERR_CUDA;
  return status_of_bits(bits);
}

const char* rl_status_string(rl_status status) {
  switch (status) {
    case RL_OK: return "ok";
    case RL_ERR_INVALID_ARG: return "invalid argument";
    case RL_ERR_UNSUPPORTED: return "unsupported configuration";
    case RL_ERR_WORKSPACE_TOO_SMALL: return "workspace too small";
    case RL_ERR_CUDA: return "CUDA runtime error";
    case RL_ERR_TARGET_OUT_OF_RANGE: return "target id outside [0, vocab)";
    case RL_ERR_GROUP_OUT_OF_RANGE: return "group id outside [0, n_groups)";
    case RL_ERR_BAD_SEQLENS: return "cu_seqlens not non-decreasing from 0 to n_rows";
    case RL_ERR_DEVICE_TIMEOUT: return "a bounded wait inside a kernel timed out";
    case RL_ERR_TOPK_ID_OUT_OF_RANGE: return "top-K OPD candidate id outside [0, vocab)";
  }
  return "unknown status";
}

rl_status rl_set_sweep_events(void* begin_event, void* end_event) {
  t_ev_begin = static_cast<cudaEvent_t>(begin_event);
  t_ev_end = static_cast<cudaEvent_t>(end_event);
  return RL_OK;
}

rl_status rl_launch_overrides_init(rl_launch_overrides* o) {
  if (!o) return RL_ERR_INVALID_ARG;
  o->sweep_kernel = o->cluster_size = o->cluster_stages = o->cluster_threads = -1;
  o->cluster_ctas_per_sm = o->stream_chunk_bytes = o->stream_slots = o->stream_hold = -1;
  o->stream_split_first = o->stream_prefetch_bytes = o->stream_ctas_per_sm = -1;
  o->stall_first_wait_ns = -1;
  o->stream_cluster = -1;
  return RL_OK;
}

rl_status rl_set_launch_overrides(const rl_launch_overrides* o) {
  rl_launch_overrides v;
  rl_launch_overrides_init(&v);
  if (o) {
    auto in = [](int32_t x, int32_t lo, int32_t hi) { return x == -1 || (x >= lo && x <= hi); };
    if (!in(o->sweep_kernel, 0, 1) || !in(o->cluster_size, 1, kMaxCluster) ||
        !in(o->cluster_stages, 1, kMaxStages) || !in(o->cluster_threads, 256, 512) ||
        !in(o->cluster_ctas_per_sm, 1, 8) || !in(o->stream_chunk_bytes, 1024, 131072) ||
        !in(o->stream_slots, 1, kMaxSlots) || !in(o->stream_hold, 0, kMaxSlots) ||
        !in(o->stream_split_first, 0, 1) || !in(o->stream_prefetch_bytes, 0, 1 << 20) ||
        (o->stream_prefetch_bytes > 0 && o->stream_prefetch_bytes % 16) ||
        (o->stream_ctas_per_sm != -1 && o->stream_ctas_per_sm != 1 &&
         o->stream_ctas_per_sm != 2 && o->stream_ctas_per_sm != 4) ||
        o->stall_first_wait_ns < -1 ||
        o->stall_first_wait_ns > 10000000000LL ||
        (o->stream_cluster != -1 && o->stream_cluster != 1 && o->stream_cluster != 2 &&
         o->stream_cluster != 4 && o->stream_cluster != 8))
      return RL_ERR_INVALID_ARG;
    v = *o;
  }
  std::lock_guard<std::mutex> lk(g_ov_mu);
  g_ov = v;
  return RL_OK;
}

int32_t rl_loss_abi_version(void) { return 131; }

}  // extern "C"

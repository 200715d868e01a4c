// Advantages of the configured estimator (Sec. 3.4: GRPO, GSPO, REINFORCE++
// plain and baseline-relative), the per-row advantage with the one-sample
// on-policy-distillation shaping (Sec. 5.2), the masked token count N, the
// training tokens of every trajectory, and validation of group ids and row
// offsets.
//
// One CTA of 1024 threads does all of it: the inputs are a few KB of
// per-trajectory data plus one byte and one float per row. Row offsets,
// per-trajectory counts and advantages are staged in shared memory when they
// fit. The row passes go one warp per trajectory over its contiguous rows.
// Every floating-point sum runs in a fixed order (lane-strided partial sums,
// xor-butterfly merges) in double precision and every count is an integer, so
// results are bit-for-bit reproducible.
#include "common.cuh"
#include "kernels.h"

namespace milesloss {

namespace {

constexpr int kWarps = kAdvThreads / 32;

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ double warp_max(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmax(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ double warp_min(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmin(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Block-wide sums in a fixed order (valid in every thread).
__device__ double block_sum(double v, double* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  double t = 0.0;
  for (int w = 0; w < kWarps; ++w) t += sh[w];
  return t;
}
// Exact integer block sum (valid in every thread).
__device__ unsigned long long block_sum_u(unsigned long long v, unsigned long long* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  unsigned long long t = 0;
  for (int w = 0; w < kWarps; ++w) t += sh[w];
  return t;
}
__device__ double block_max(double v, double* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_max(v);
  __syncthreads();
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  double t = -INFINITY;
  for (int w = 0; w < kWarps; ++w) t = fmax(t, sh[w]);
  return t;
}

// The statistics of group g, computed by one warp that scans the group ids
// for the group's members: n, mean, the standard deviation with its floor,
// and whether all rewards are equal. In double precision.
__device__ void group_stats(const AdvArgs& a, const int* gid, const float* rew, int g, int lane) {
  WsPtrs ws = a.ws;
  int n = 0;
  double sum = 0.0, wmax = -INFINITY, wmin = INFINITY;
#pragma unroll 4
  for (int i = lane; i < a.n_traj; i += 32) {
    if (gid[i] == g) {
      const double w = rew[i];
      ++n;
      sum += w;
      wmax = fmax(wmax, w);
      wmin = fmin(wmin, w);
    }
  }
  n = warp_sum_i(n);
  sum = warp_sum(sum);
  wmax = warp_max(wmax);
  wmin = warp_min(wmin);
  const double mu = n > 0 ? sum / n : 0.0;
  double ss = 0.0;
#pragma unroll 4
  for (int i = lane; i < a.n_traj; i += 32) {
    if (gid[i] == g) {
      const double d = static_cast<double>(rew[i]) - mu;
      ss += d * d;
    }
  }
  ss = warp_sum(ss);
  // A group whose rewards are all equal (this includes one-member groups)
  // carries no advantage signal: its GRPO advantages are exactly zero.
  const int flat = (n == 0) || (wmax == wmin);
  double den = 1.0;
  if (a.normalize_std && !flat) {
    const int ddof = a.unbiased_std ? 1 : 0;
    den = fmax(sqrt(ss / static_cast<double>(n - ddof)), static_cast<double>(a.std_floor));
  }
  if (lane == 0) {
    ws.g_mu[g] = mu;
    ws.g_den[g] = den;
    ws.g_flag[g] = flat;
    if (a.group_sizes) a.group_sizes[g] = n;
  }
}

// Group statistics for calls with more than kInlineGroups groups, one
// 32-thread block per group. GB300 runs double precision at a small fraction
// of its fp32 rate: spread over the SMs, the groups' double arithmetic no
// longer queues on the one SM that runs k_advantages.
__global__ void __launch_bounds__(32) k_groups(const AdvArgs a) {
  for (int g = blockIdx.x; g < a.n_groups; g += gridDim.x)
    group_stats(a, a.gid, a.rewards, g, threadIdx.x);
}

__global__ void __launch_bounds__(kAdvThreads, 1) k_advantages(const AdvArgs a) {
  extern __shared__ __align__(16) int dyn[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __shared__ unsigned int s_err;
  __shared__ double s_red[kWarps];
  __shared__ unsigned long long s_cnt[kWarps];
  WsPtrs ws = a.ws;
  // Shared copies, when they fit, of cu (n_traj + 1), the per-trajectory
  // token counts and advantages, group ids and rewards (n_traj each).
  const bool on_chip = a.smem_traj;
  const int nt = a.n_traj;
  int* cu = on_chip ? dyn : const_cast<int*>(a.cu);
  int* cnt_i = on_chip ? dyn + (nt + 1) : ws.traj_n;
  const int* gid = on_chip ? dyn + (3 * nt + 1) : a.gid;
  const float* rew = on_chip ? reinterpret_cast<const float*>(dyn + (4 * nt + 1)) : a.rewards;
  if (tid == 0) {
    s_err = 0;
    ws.hdr->err_bits = 0;
    ws.hdr->ticket = 0;
  }
  for (int i = tid; i <= nt; i += kAdvThreads) {
    if (on_chip) {
      cu[i] = a.cu[i];
      if (i < nt) {
        dyn[3 * nt + 1 + i] = a.gid[i];
        reinterpret_cast<float*>(dyn + 4 * nt + 1)[i] = a.rewards[i];
      }
    }
    if (i < nt) cnt_i[i] = 0;
  }
  __syncthreads();

  // ---- validation
  unsigned int err = 0;
  for (int i = tid; i < a.n_traj; i += kAdvThreads) {
    if (cu[i] > cu[i + 1]) err |= kErrSeqlens;
    const int g = gid[i];
    if (g < 0 || g >= a.n_groups) err |= kErrGroup;
  }
  if (tid == 0 && (cu[0] != 0 || static_cast<long long>(cu[a.n_traj]) != a.R_total))
    err |= kErrSeqlens;
  if (err) atomicOr(&s_err, err);

  // ---- group statistics: one warp per group here when there are few
  // (otherwise k_groups computed them just before)
  if (a.n_groups <= kInlineGroups)
    for (int g = warp; g < a.n_groups; g += kWarps) group_stats(a, gid, rew, g, lane);
  __syncthreads();
  const bool cu_ok = (s_err & kErrSeqlens) == 0;
  const bool rpp = a.estimator == RL_EST_REINFORCEPP || a.estimator == RL_EST_REINFORCEPP_BASELINE;

  // ---- per-trajectory base value (kept in double in a register-free way:
  // recomputed from the group table where needed)
  auto base_value = [&](int i) -> double {
    const int g = gid[i];
    const bool gok = g >= 0 && g < a.n_groups;
    const double w = rew[i];
    if (a.estimator == RL_EST_REINFORCEPP) return w;
    if (a.estimator == RL_EST_REINFORCEPP_BASELINE) return gok ? w - ws.g_mu[g] : 0.0;
    if (!gok || ws.g_flag[g]) return 0.0;  // GRPO, GSPO
    return (w - ws.g_mu[g]) / ws.g_den[g];
  };

  // Trajectory advantages (in shared memory when the trajectory tables fit).
  float* a_s = on_chip ? reinterpret_cast<float*>(dyn + 2 * a.n_traj + 1) : ws.a_traj;
  auto publish = [&](int i, double A) {
    a_s[i] = static_cast<float>(A);
    if (on_chip) ws.a_traj[i] = static_cast<float>(A);
    if (a.advantages) a.advantages[i] = static_cast<float>(A);
  };
  // GRPO and GSPO: the trajectory advantage is final before any row is read,
  // so one pass over the rows counts and writes the row advantages.
  if (!rpp) {
    for (int i = tid; i < a.n_traj; i += kAdvThreads) publish(i, base_value(i));
    __syncthreads();
  }

  // ---- passes over the rows, one warp per trajectory (its rows are the
  // contiguous range [cu[i], cu[i+1]); several warps per trajectory when
  // there are fewer trajectories than warps): the lanes count the trajectory's
  // training tokens from 16-byte blocks of the mask and fill its row
  // advantages with 16-byte stores, with the one-sample OPD shaping. With
  // invalid row offsets every row gets advantage 0 (plus the shaping) and
  // only N is counted, row by row. A shard sees the part of each trajectory
  // that falls in its rows [row0, row0 + R) (local indices from 0); given the
  // counts of every shard (counts_in), it takes N and the trajectories'
  // counts from them instead of counting.
  const bool lookup = cu_ok && a.n_traj > 0;
  const bool mask_vec = (reinterpret_cast<uintptr_t>(a.mask) & 15u) == 0;
  const bool row_vec = (reinterpret_cast<uintptr_t>(ws.a_row) & 15u) == 0;
  const bool opd_vec = a.teacher && ((reinterpret_cast<uintptr_t>(a.rho) |
                                      reinterpret_cast<uintptr_t>(a.teacher)) & 15u) == 0;
  auto opd = [&](long long t) { return a.teacher ? a.opd_coef * (a.rho[t] - a.teacher[t]) : 0.0f; };
  // trajectory i's rows in this call, as local indices [lo, hi)
  auto local_lo = [&](int i) { return max(static_cast<long long>(cu[i]), a.row0) - a.row0; };
  auto local_hi = [&](int i) {
    return max(min(static_cast<long long>(cu[i + 1]), a.row0 + a.R) - a.row0, local_lo(i));
  };
  // With fewer trajectories than warps, wpt warps share each trajectory
  // (warp `sub` of them takes every wpt-th 512-row or 128-row piece).
  const int wpt = a.n_traj > 0 ? max(1, kWarps / a.n_traj) : 1;
  const int traj_groups = kWarps / wpt;
  const int group = warp / wpt, sub = warp % wpt;
  auto count_rows = [&](long long lo, long long hi) {  // training tokens in [lo, hi), warp-wide
    int c = 0;
    for (long long b = (lo & ~15LL) + 16LL * (lane + 32 * sub); b < hi; b += 16LL * 32 * wpt) {
      if (mask_vec && b >= lo && b + 16 <= hi) {
        const uint4 v = *reinterpret_cast<const uint4*>(a.mask + b);
        c += (__popc(__vcmpne4(v.x, 0u)) + __popc(__vcmpne4(v.y, 0u)) +
              __popc(__vcmpne4(v.z, 0u)) + __popc(__vcmpne4(v.w, 0u))) >> 3;
      } else {
        for (long long t = max(b, lo); t < min(b + 16, hi); ++t) c += a.mask[t] != 0;
      }
    }
    return warp_sum_i(c);
  };
  auto write_rows = [&](long long lo, long long hi, float A) {  // row advantages of [lo, hi)
    for (long long b = (lo & ~3LL) + 4LL * (lane + 32 * sub); b < hi; b += 4LL * 32 * wpt) {
      if (row_vec && b >= lo && b + 4 <= hi && (!a.teacher || opd_vec)) {
        float4 v = make_float4(A, A, A, A);
        if (a.teacher) {
          const float4 r = *reinterpret_cast<const float4*>(a.rho + b);
          const float4 q = *reinterpret_cast<const float4*>(a.teacher + b);
          v.x -= a.opd_coef * (r.x - q.x);
          v.y -= a.opd_coef * (r.y - q.y);
          v.z -= a.opd_coef * (r.z - q.z);
          v.w -= a.opd_coef * (r.w - q.w);
        }
        *reinterpret_cast<float4*>(ws.a_row + b) = v;
      } else {
        for (long long t = max(b, lo); t < min(b + 4, hi); ++t) ws.a_row[t] = A - opd(t);
      }
    }
  };
  unsigned long long n_tok = 0;
  if (lookup && a.counts_in) {
    for (int i = tid; i < a.n_traj; i += kAdvThreads) {
      const int c = a.counts_in[i];
      cnt_i[i] = c;
      n_tok += static_cast<unsigned long long>(c);
    }
    if (!rpp && group < traj_groups)
      for (int i = group; i < a.n_traj; i += traj_groups) write_rows(local_lo(i), local_hi(i), a_s[i]);
    __syncthreads();
  } else if (lookup) {
    if (group < traj_groups) {
      for (int i = group; i < a.n_traj; i += traj_groups) {
        const long long lo = local_lo(i), hi = local_hi(i);
        const int c = count_rows(lo, hi);
        if (lane == 0 && c) {
          atomicAdd(&cnt_i[i], c);  // integer: exact in any order
          n_tok += static_cast<unsigned long long>(c);
        }
        if (!rpp) write_rows(lo, hi, a_s[i]);
      }
    }
    __syncthreads();  // every trajectory's count complete
    if (a.counts_out)
      for (int i = tid; i < a.n_traj; i += kAdvThreads) a.counts_out[i] = cnt_i[i];
  } else {
    for (long long t = tid; t < a.R; t += kAdvThreads) {
      n_tok += a.mask[t] != 0;
      if (!rpp) ws.a_row[t] = -opd(t);
    }
  }
  const double N = static_cast<double>(block_sum_u(n_tok, s_cnt));

  // ---- REINFORCE++: normalise the returns over the training tokens, then
  // a second pass writes the row advantages
  if (rpp) {
    double sb = 0.0, bmax = -INFINITY, bmin = INFINITY;
    for (int i = tid; i < a.n_traj; i += kAdvThreads) {
      const int n_i = cnt_i[i];
      if (n_i == 0) continue;
      const double b = base_value(i);
      sb += b * n_i;
      bmax = fmax(bmax, b);
      bmin = fmin(bmin, b);
    }
    sb = block_sum(sb, s_red);
    bmax = block_max(bmax, s_red);
    bmin = -block_max(-bmin, s_red);
    const bool zero_all = !(N > 0.0) || !(bmax != bmin);
    const double mu = N > 0.0 ? sb / N : 0.0;
    double ss = 0.0;
    for (int i = tid; i < a.n_traj; i += kAdvThreads) {
      const int n_i = cnt_i[i];
      if (n_i == 0) continue;
      const double d = base_value(i) - mu;
      ss += d * d * n_i;
    }
    ss = block_sum(ss, s_red);
    double den = 1.0;
    if (a.normalize_std) {
      const double ddof = a.unbiased_std ? 1.0 : 0.0;
      const double var = N > ddof ? ss / (N - ddof) : 0.0;
      den = fmax(sqrt(var), static_cast<double>(a.std_floor));
    }
    for (int i = tid; i < a.n_traj; i += kAdvThreads)
      publish(i, zero_all ? 0.0 : (base_value(i) - mu) / den);
    __syncthreads();
    if (lookup) {
      if (group < traj_groups)
        for (int i = group; i < a.n_traj; i += traj_groups)
          write_rows(local_lo(i), local_hi(i), a_s[i]);
    } else {
      for (long long t = tid; t < a.R; t += kAdvThreads) ws.a_row[t] = -opd(t);
    }
  }

  // ---- the training tokens of each trajectory, and how many trajectories train
  int n_seq = 0;
  for (int i = tid; i < a.n_traj; i += kAdvThreads) {
    const int n_i = cnt_i[i];
    if (on_chip) ws.traj_n[i] = n_i;
    n_seq += (n_i > 0);
  }
  const unsigned long long n_seq_all = block_sum_u(static_cast<unsigned long long>(n_seq), s_cnt);
  if (tid == 0) {
    ws.hdr->n_tokens = static_cast<long long>(N);
    ws.hdr->n_seq = static_cast<long long>(n_seq_all);  // exact integer counts
    if (s_err) atomicOr(&ws.hdr->err_bits, s_err);
  }
}

}  // namespace

const void* adv_kernel() { return reinterpret_cast<const void*>(&k_advantages); }
const void* groups_kernel() { return reinterpret_cast<const void*>(&k_groups); }

}  // namespace milesloss

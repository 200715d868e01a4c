// Advantages of the configured estimator (Sec. 3.4: GRPO, GSPO, REINFORCE++
// plain and baseline-relative), the per-row advantage with the one-sample
// on-policy-distillation shaping (Sec. 5.2), the masked token count N, the
// training tokens of every trajectory, and validation of group ids and row
// offsets.
//
// One CTA of 1024 threads does all of it: the inputs are a few KB of
// per-trajectory data plus one byte and one float per row. Row offsets and
// per-trajectory counts are staged in shared memory when they fit, so the
// per-row trajectory lookup (a binary search) stays on chip. Every sum runs
// in a fixed order (lane-strided partial sums, xor-butterfly merges) in
// double precision, so results are bit-for-bit reproducible.
#include "common.cuh"
#include "kernels.h"

namespace milesloss {

namespace {

constexpr int kWarps = kAdvThreads / 32;
constexpr int kRowBlock = 16;  // consecutive rows per thread in the row passes

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

// Trajectory of row t: the last i with cu[i] <= t (cu valid: cu[0] = 0 <= t < cu[n]).
__device__ __forceinline__ int traj_of(const int* cu, int n_traj, long long t) {
  int lo = 0, hi = n_traj;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (static_cast<long long>(cu[mid]) <= t) lo = mid; else hi = mid;
  }
  return lo;
}

__global__ void __launch_bounds__(kAdvThreads, 1) k_advantages(const AdvArgs a) {
  extern __shared__ __align__(16) int dyn[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __shared__ unsigned int s_err;
  __shared__ double s_red[kWarps];
  __shared__ unsigned long long s_cnt[kWarps];
  WsPtrs ws = a.ws;
  // shared copies of cu (n_traj + 1) and the per-trajectory token counts
  const bool on_chip = a.smem_traj;
  int* cu = on_chip ? dyn : const_cast<int*>(a.cu);
  int* cnt_i = on_chip ? dyn + (a.n_traj + 1) : ws.traj_n;
  if (tid == 0) {
    s_err = 0;
    ws.hdr->err_bits = 0;
    ws.hdr->ticket = 0;
  }
  for (int i = tid; i <= a.n_traj; i += kAdvThreads) {
    if (on_chip) cu[i] = a.cu[i];
    if (i < a.n_traj) cnt_i[i] = 0;
  }
  __syncthreads();

  // ---- validation
  unsigned int err = 0;
  for (int i = tid; i < a.n_traj; i += kAdvThreads) {
    if (cu[i] > cu[i + 1]) err |= kErrSeqlens;
    const int g = a.gid[i];
    if (g < 0 || g >= a.n_groups) err |= kErrGroup;
  }
  if (tid == 0 && (cu[0] != 0 || static_cast<long long>(cu[a.n_traj]) != a.R)) err |= kErrSeqlens;
  if (err) atomicOr(&s_err, err);

  // ---- group statistics: one warp per group, members found by scanning.
  for (int g = warp; g < a.n_groups; g += kWarps) {
    int n = 0;
    double sum = 0.0, wmax = -INFINITY, wmin = INFINITY;
    for (int i = lane; i < a.n_traj; i += 32) {
      if (a.gid[i] == g) {
        const double w = a.rewards[i];
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
    for (int i = lane; i < a.n_traj; i += 32) {
      if (a.gid[i] == g) {
        const double d = static_cast<double>(a.rewards[i]) - mu;
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
  __syncthreads();
  const bool cu_ok = (s_err & kErrSeqlens) == 0;
  const bool rpp = a.estimator == RL_EST_REINFORCEPP || a.estimator == RL_EST_REINFORCEPP_BASELINE;

  // ---- per-trajectory base value (kept in double in a register-free way:
  // recomputed from the group table where needed)
  auto base_value = [&](int i) -> double {
    const int g = a.gid[i];
    const bool gok = g >= 0 && g < a.n_groups;
    const double w = a.rewards[i];
    if (a.estimator == RL_EST_REINFORCEPP) return w;
    if (a.estimator == RL_EST_REINFORCEPP_BASELINE) return gok ? w - ws.g_mu[g] : 0.0;
    if (!gok || ws.g_flag[g]) return 0.0;  // GRPO, GSPO
    return (w - ws.g_mu[g]) / ws.g_den[g];
  };

  // ---- per-row pass 1: N, and (for the estimators that use them) the
  // training tokens of each trajectory. Consecutive rows mostly share a
  // trajectory, so the lanes of a warp that do add once per trajectory.
  // Each thread takes blocks of kRowBlock consecutive rows (one 16-byte load
  // of the mask when the block is whole and aligned), so that the loads of a
  // pass are few and independent.
  const bool need_counts = rpp || a.estimator == RL_EST_GSPO;
  const bool lookup = cu_ok && a.n_traj > 0;
  const bool mask_vec = (reinterpret_cast<uintptr_t>(a.mask) & 15u) == 0;
  unsigned long long n_tok = 0;
  for (long long b0 = static_cast<long long>(tid) * kRowBlock; b0 < a.R;
       b0 += static_cast<long long>(kAdvThreads) * kRowBlock) {
    const int nb = static_cast<int>(min(static_cast<long long>(kRowBlock), a.R - b0));
    // the block's mask bytes, packed four to a register (byte j in word j / 4)
    uint32_t m[kRowBlock / 4];
    if (nb == kRowBlock && mask_vec) {
      const uint4 v = *reinterpret_cast<const uint4*>(a.mask + b0);
      m[0] = v.x; m[1] = v.y; m[2] = v.z; m[3] = v.w;
    } else {
#pragma unroll
      for (int q = 0; q < kRowBlock / 4; ++q) m[q] = 0u;
      for (int j = 0; j < nb; ++j)
        m[j >> 2] |= (a.mask[b0 + j] != 0 ? 1u : 0u) << (8 * (j & 3));
    }
    int i = (need_counts && lookup) ? traj_of(cu, a.n_traj, b0) : 0;
    int run = 0;
#pragma unroll
    for (int j = 0; j < kRowBlock; ++j) {
      if (j >= nb) break;
      const bool tr = ((m[j >> 2] >> (8 * (j & 3))) & 0xffu) != 0;
      n_tok += tr;
      if (need_counts && lookup) {
        while (i + 1 < a.n_traj && cu[i + 1] <= b0 + j) {  // next trajectory
          if (run) atomicAdd(&cnt_i[i], run);
          run = 0;
          ++i;
        }
        run += tr;
      }
    }
    if (need_counts && lookup && run) atomicAdd(&cnt_i[i], run);
  }
  const double N = static_cast<double>(block_sum_u(n_tok, s_cnt));

  // ---- REINFORCE++: normalise the returns over the training tokens
  double mu = 0.0, den = 1.0;
  bool zero_all = false;
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
    zero_all = !(N > 0.0) || !(bmax != bmin);
    mu = N > 0.0 ? sb / N : 0.0;
    double ss = 0.0;
    for (int i = tid; i < a.n_traj; i += kAdvThreads) {
      const int n_i = cnt_i[i];
      if (n_i == 0) continue;
      const double d = base_value(i) - mu;
      ss += d * d * n_i;
    }
    ss = block_sum(ss, s_red);
    if (a.normalize_std) {
      const double ddof = a.unbiased_std ? 1.0 : 0.0;
      const double var = N > ddof ? ss / (N - ddof) : 0.0;
      den = fmax(sqrt(var), static_cast<double>(a.std_floor));
    }
  }

  // ---- per-trajectory advantage and the count of trajectories that train
  int n_seq = 0;
  for (int i = tid; i < a.n_traj; i += kAdvThreads) {
    double A = base_value(i);
    if (rpp) A = zero_all ? 0.0 : (A - mu) / den;
    ws.a_traj[i] = static_cast<float>(A);
    if (a.advantages) a.advantages[i] = static_cast<float>(A);
    const int n_i = cnt_i[i];
    if (on_chip) ws.traj_n[i] = n_i;
    n_seq += (n_i > 0);
  }
  const unsigned long long n_seq_all = block_sum_u(static_cast<unsigned long long>(n_seq), s_cnt);

  // ---- per-row pass 2: the row's advantage, with the one-sample OPD shaping.
  // The trajectory's advantage is reloaded only when a block crosses into the
  // next trajectory, and a whole aligned block leaves in four 16-byte stores.
  const bool row_vec = (reinterpret_cast<uintptr_t>(ws.a_row) & 15u) == 0;
  for (long long b0 = static_cast<long long>(tid) * kRowBlock; b0 < a.R;
       b0 += static_cast<long long>(kAdvThreads) * kRowBlock) {
    const int nb = static_cast<int>(min(static_cast<long long>(kRowBlock), a.R - b0));
    int i = lookup ? traj_of(cu, a.n_traj, b0) : 0;
    float A_i = lookup ? ws.a_traj[i] : 0.0f;
    float out[kRowBlock];
#pragma unroll
    for (int j = 0; j < kRowBlock; ++j) {
      if (lookup && j < nb && i + 1 < a.n_traj && cu[i + 1] <= b0 + j) {
        do { ++i; } while (i + 1 < a.n_traj && cu[i + 1] <= b0 + j);  // next trajectory
        A_i = ws.a_traj[i];
      }
      out[j] = A_i;
    }
    if (a.teacher) {
#pragma unroll
      for (int j = 0; j < kRowBlock; ++j)
        if (j < nb) out[j] -= a.opd_coef * (a.rho[b0 + j] - a.teacher[b0 + j]);
    }
    if (nb == kRowBlock && row_vec) {
      float4* dst = reinterpret_cast<float4*>(ws.a_row + b0);
#pragma unroll
      for (int q = 0; q < kRowBlock / 4; ++q)
        dst[q] = make_float4(out[4 * q], out[4 * q + 1], out[4 * q + 2], out[4 * q + 3]);
    } else {
#pragma unroll
      for (int j = 0; j < kRowBlock; ++j)
        if (j < nb) ws.a_row[b0 + j] = out[j];
    }
  }
  if (tid == 0) {
    ws.hdr->n_tokens = static_cast<long long>(N);
    ws.hdr->n_seq = static_cast<long long>(n_seq_all);  // exact integer counts
    if (s_err) atomicOr(&ws.hdr->err_bits, s_err);
  }
}

}  // namespace

const void* adv_kernel() { return reinterpret_cast<const void*>(&k_advantages); }

}  // namespace milesloss

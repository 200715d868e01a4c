// Group-relative advantages (GRPO, Sec. 2 and Sec. 9.1), the per-row
// advantage with optional on-policy-distillation shaping (Sec. 5.2), the
// masked token count N, and validation of group ids and row offsets.
//
// One CTA of 1024 threads does all of it; the inputs are a few KB of
// per-trajectory data plus one byte and one float per row, so the kernel
// is a small fraction of a call. Every sum runs in a fixed order (lane-
// strided partial sums, xor-butterfly merges), so results are bit-for-bit
// reproducible, and all statistics are accumulated in double precision.
#include "common.cuh"
#include "kernels.h"

namespace milesloss {

namespace {

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

__global__ void __launch_bounds__(kAdvThreads, 1) k_advantages(const AdvArgs a) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int kWarps = kAdvThreads / 32;
  __shared__ unsigned int s_err;
  __shared__ unsigned long long s_cnt[kWarps];
  WsPtrs ws = a.ws;
  if (tid == 0) {
    s_err = 0;
    ws.hdr->err_bits = 0;
    ws.hdr->ticket = 0;
  }
  __syncthreads();

  // ---- validation
  unsigned int err = 0;
  for (int i = tid; i < a.n_traj; i += kAdvThreads) {
    if (a.cu[i] > a.cu[i + 1]) err |= kErrSeqlens;
    const int g = a.gid[i];
    if (g < 0 || g >= a.n_groups) err |= kErrGroup;
  }
  if (tid == 0 && (a.cu[0] != 0 || static_cast<long long>(a.cu[a.n_traj]) != a.R))
    err |= kErrSeqlens;
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
    // carries no advantage signal: its advantages are exactly zero.
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

  // ---- per-trajectory advantage
  for (int i = tid; i < a.n_traj; i += kAdvThreads) {
    const int g = a.gid[i];
    double A = 0.0;
    if (g >= 0 && g < a.n_groups && !ws.g_flag[g])
      A = (static_cast<double>(a.rewards[i]) - ws.g_mu[g]) / ws.g_den[g];
    ws.a_traj[i] = static_cast<float>(A);
    if (a.advantages) a.advantages[i] = static_cast<float>(A);
  }
  __syncthreads();
  const bool cu_ok = (s_err & kErrSeqlens) == 0;

  // ---- per-row advantage (trajectory of row t: last i with cu[i] <= t) and N
  unsigned long long cnt = 0;
  for (long long t = tid; t < a.R; t += kAdvThreads) {
    float A = 0.0f;
    if (cu_ok && a.n_traj > 0) {
      int lo = 0, hi = a.n_traj;  // invariant: cu[lo] <= t < cu[hi]
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (static_cast<long long>(a.cu[mid]) <= t) lo = mid; else hi = mid;
      }
      A = ws.a_traj[lo];
    }
    if (a.teacher) A -= a.opd_coef * (a.rho[t] - a.teacher[t]);
    ws.a_row[t] = A;
    cnt += (a.mask[t] != 0);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  if (lane == 0) s_cnt[warp] = cnt;
  __syncthreads();
  if (tid == 0) {
    unsigned long long N = 0;
    for (int w = 0; w < kWarps; ++w) N += s_cnt[w];
    ws.hdr->n_tokens = static_cast<long long>(N);
    if (s_err) atomicOr(&ws.hdr->err_bits, s_err);
  }
}

}  // namespace

const void* adv_kernel() { return reinterpret_cast<const void*>(&k_advantages); }

}  // namespace milesloss

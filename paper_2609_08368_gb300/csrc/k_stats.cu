// The masked token-mean of the loss and the reported metrics: means over
// training tokens of the PG term, k3, entropy, ratio, |r - 1|, |logp -
// rollout logp| (the train/rollout divergence of Sec. 9.2) and the
// correction ratio (Sec. 3.4), min / max ratio, and exact clip counts.
//
// Each block reduces a fixed strided set of rows into partial sums
// (butterfly merges in a fixed order), stores them in the workspace, and the
// last block to finish (an atomic ticket, no waiting) merges the partials in
// double precision in block order. The grid size depends only on the row
// count, so the scalar loss is bit-for-bit reproducible.
#include "common.cuh"
#include "kernels.h"

namespace milesloss {

namespace {

// Per-block partial sums: fp32 within a block (a fixed-order tree over at
// most kStatThreads rows; its rounding is far below the statistics'
// tolerance), exact integer counts; the last block merges the partials in
// double precision.
struct Part {
  float v[9];  // ell, pg, k3, H, r, |r-1|, |logp-rho|, rc, |rc-1|
  float rmin, rmax;
  unsigned int c[5];  // n, clip_hi, clip_lo, dual, corr_clip
};

__device__ __forceinline__ void part_zero(Part& p) {
#pragma unroll
  for (int i = 0; i < 9; ++i) p.v[i] = 0.0f;
  p.rmin = INFINITY;
  p.rmax = -INFINITY;
#pragma unroll
  for (int i = 0; i < 5; ++i) p.c[i] = 0u;
}

__device__ __forceinline__ void part_merge_shfl(Part& p, int o) {
#pragma unroll
  for (int i = 0; i < 9; ++i) p.v[i] += __shfl_xor_sync(0xffffffffu, p.v[i], o);
  p.rmin = fminf(p.rmin, __shfl_xor_sync(0xffffffffu, p.rmin, o));
  p.rmax = fmaxf(p.rmax, __shfl_xor_sync(0xffffffffu, p.rmax, o));
#pragma unroll
  for (int i = 0; i < 5; ++i) p.c[i] += __shfl_xor_sync(0xffffffffu, p.c[i], o);
}

// Block reduction in a fixed order; the result is valid in thread 0.
__device__ void block_reduce(Part& p, Part* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  constexpr int kWarps = kStatThreads / 32;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) part_merge_shfl(p, o);
  if (lane == 0) sh[warp] = p;
  __syncthreads();
  if (warp == 0) {
    if (lane < kWarps) p = sh[lane]; else part_zero(p);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part_merge_shfl(p, o);
  }
}

__device__ __forceinline__ void to_stat(const Part& p, StatPart& s) {
  s.s_ell = p.v[0]; s.s_pg = p.v[1]; s.s_k3 = p.v[2]; s.s_H = p.v[3]; s.s_r = p.v[4];
  s.s_rabs = p.v[5]; s.s_lpabs = p.v[6]; s.s_rc = p.v[7]; s.s_rcabs = p.v[8];
  s.rmin = p.rmin; s.rmax = p.rmax;
  s.n = p.c[0]; s.n_hi = p.c[1]; s.n_lo = p.c[2]; s.n_dual = p.c[3]; s.n_corr = p.c[4];
}

// The final merge, in double precision: one partial per thread, then a
// fixed-order tree.
struct Final {
  double v[9];
  float rmin, rmax;
  unsigned long long c[5];
};

__device__ __forceinline__ void final_load(const StatPart* sp, Final& f) {
  const double* d = reinterpret_cast<const double*>(sp);
#pragma unroll
  for (int i = 0; i < 9; ++i) f.v[i] = __ldcg(d + i);
  f.rmin = __ldcg(&sp->rmin);
  f.rmax = __ldcg(&sp->rmax);
  const unsigned long long* c = &sp->n;
#pragma unroll
  for (int i = 0; i < 5; ++i) f.c[i] = __ldcg(c + i);
}

__device__ __forceinline__ void final_zero(Final& f) {
#pragma unroll
  for (int i = 0; i < 9; ++i) f.v[i] = 0.0;
  f.rmin = INFINITY;
  f.rmax = -INFINITY;
#pragma unroll
  for (int i = 0; i < 5; ++i) f.c[i] = 0ull;
}

__device__ __forceinline__ void final_merge_shfl(Final& f, int o) {
#pragma unroll
  for (int i = 0; i < 9; ++i) f.v[i] += __shfl_xor_sync(0xffffffffu, f.v[i], o);
  f.rmin = fminf(f.rmin, __shfl_xor_sync(0xffffffffu, f.rmin, o));
  f.rmax = fmaxf(f.rmax, __shfl_xor_sync(0xffffffffu, f.rmax, o));
#pragma unroll
  for (int i = 0; i < 5; ++i) f.c[i] += __shfl_xor_sync(0xffffffffu, f.c[i], o);
}

// Means over the n = c[0] training tokens; zeros when there are none.
__device__ rl_loss_stats stats_of(const double* v, const unsigned long long* c, float rmin,
                                  float rmax) {
  rl_loss_stats o;
  const unsigned long long n = c[0];
  const double inv = n ? 1.0 / static_cast<double>(n) : 0.0;
  o.loss = v[0] * inv;
  o.pg_loss_mean = v[1] * inv;
  o.kl_mean = v[2] * inv;
  o.entropy_mean = v[3] * inv;
  o.ratio_mean = v[4] * inv;
  o.ratio_absdev_mean = v[5] * inv;
  o.logprob_absdiff_mean = v[6] * inv;
  o.corr_ratio_mean = v[7] * inv;
  o.corr_absdev_mean = v[8] * inv;
  o.ratio_min = n ? rmin : 0.0f;
  o.ratio_max = n ? rmax : 0.0f;
  o.n_tokens = static_cast<int64_t>(n);
  o.n_clip_hi = static_cast<int64_t>(c[1]);
  o.n_clip_lo = static_cast<int64_t>(c[2]);
  o.n_dual_clip = static_cast<int64_t>(c[3]);
  o.n_corr_clip = static_cast<int64_t>(c[4]);
  return o;
}

__global__ void __launch_bounds__(kStatThreads) k_stats(const StatArgs a) {
  __shared__ Part sh[kStatThreads / 32];
  __shared__ Final shf[kStatThreads / 32];
  __shared__ int s_last;
  WsPtrs ws = a.ws;
  Part p;
  part_zero(p);
  const long long stride = static_cast<long long>(gridDim.x) * kStatThreads;
  for (long long t = blockIdx.x * static_cast<long long>(kStatThreads) + threadIdx.x; t < a.R;
       t += stride) {
    if (!a.mask[t]) continue;
    const uint8_t f = ws.flags[t];
    const float r = ws.r[t], rc = ws.rc[t];
    p.v[0] += ws.ell[t];
    p.v[1] += ws.pg[t];
    p.v[2] += ws.k3[t];
    p.v[3] += ws.H[t];
    p.v[4] += r;
    p.v[5] += fabsf(r - 1.0f);
    p.v[6] += fabsf(ws.logp[t] - a.rho[t]);
    p.v[7] += rc;
    p.v[8] += fabsf(rc - 1.0f);
    p.rmin = fminf(p.rmin, r);
    p.rmax = fmaxf(p.rmax, r);
    p.c[0] += 1;
    p.c[1] += (f & kFlagClipHi) ? 1 : 0;
    p.c[2] += (f & kFlagClipLo) ? 1 : 0;
    p.c[3] += (f & kFlagDual) ? 1 : 0;
    p.c[4] += (f & kFlagCorrClip) ? 1 : 0;
  }
  block_reduce(p, sh);
  if (threadIdx.x == 0) {
    to_stat(p, ws.parts[blockIdx.x]);
    __threadfence();
    const unsigned int ticket = atomicAdd(&ws.hdr->ticket, 1u);
    s_last = (ticket == gridDim.x - 1) ? 1 : 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  // Last block: merge the partials in block order (one per thread, then a tree).
  Final fin;
  if (static_cast<int>(threadIdx.x) < static_cast<int>(gridDim.x)) final_load(&ws.parts[threadIdx.x], fin);
  else final_zero(fin);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) final_merge_shfl(fin, o);
  if (lane == 0) shf[warp] = fin;
  __syncthreads();
  if (warp == 0) {
    if (lane < kStatThreads / 32) fin = shf[lane]; else final_zero(fin);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) final_merge_shfl(fin, o);
  }
  if (threadIdx.x == 0) {
    if (a.part_out) {
      rl_loss_partials p;
      for (int i = 0; i < 9; ++i) p.sum[i] = fin.v[i];
      for (int i = 0; i < 5; ++i) p.count[i] = static_cast<double>(fin.c[i]);
      p.max[0] = fin.c[0] ? -static_cast<double>(fin.rmin) : -INFINITY;
      p.max[1] = fin.c[0] ? static_cast<double>(fin.rmax) : -INFINITY;
      *a.part_out = p;
    } else {
      *a.out = stats_of(fin.v, fin.c, fin.rmin, fin.rmax);
    }
    ws.hdr->ticket = 0;
  }
}

// The statistics of a sharded call from its shards' combined partials.
__global__ void k_finish(const FinishArgs a) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  const rl_loss_partials p = *a.part;
  unsigned long long c[5];
  for (int i = 0; i < 5; ++i) c[i] = static_cast<unsigned long long>(p.count[i]);
  *a.out = stats_of(p.sum, c, static_cast<float>(-p.max[0]), static_cast<float>(p.max[1]));
}

}  // namespace

const void* stats_kernel() { return reinterpret_cast<const void*>(&k_stats); }
const void* finish_kernel() { return reinterpret_cast<const void*>(&k_finish); }

}  // namespace milesloss

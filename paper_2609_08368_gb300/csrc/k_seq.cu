// GSPO's sequence-level objective (Sec. 3.4 lists GSPO among the shipped
// estimators): per trajectory i with n_i training tokens,
//   s_i = exp((1/n_i) sum_{t in i, m_t = 1} (logp_t - base_t)),
//   pg_i = max(-A_i s_i, -A_i clip(s_i, 1-eps_lo, 1+eps_hi)), capped at -A_i c
//          for A_i < 0 by the dual clip,
// and the policy term of the loss is the mean of pg_i over the n_seq
// trajectories that have training tokens. Written per row so that the
// masked token-mean over N tokens is that loss: a token of trajectory i
// carries l_t = (N / (n_seq n_i)) w_t pg_i + beta k3_t - gamma H_t and
//   G_t = (N / (n_seq n_i)) mean_i(w) (-A_i s_i if unclipped else 0)
//         + beta (1 - exp(q_t - logp_t)),
// w_t the token's ratio-correction weight (1 without a correction).
//
// Runs after the forward sweep (which left logp, H, k3 and the correction
// ratio of every row in the workspace) and before the gradient sweep: one
// block per trajectory, sums in a fixed order in double precision. In a
// row-sharded call a trajectory's rows may lie on several shards: each shard
// first writes its part of the two sums (sums_out), the caller adds them
// over the shards, and each shard then applies the trajectory's terms to its
// own rows from the added sums (sums_in).
#include "common.cuh"
#include "kernels.h"

namespace milesloss {

namespace {

constexpr int kThreads = kSeqThreads;
constexpr int kWarps = kThreads / 32;

__global__ void __launch_bounds__(kThreads) k_seq(const SeqArgs a) {
  __shared__ double s_a[kWarps], s_b[kWarps];
  __shared__ float s_out[4];  // s_i, scale * pg_i, scale * mean_w * (-A s_i) or 0, flags
  WsPtrs ws = a.ws;
  const int i = blockIdx.x;
  if (ws.hdr->err_bits & kErrSeqlens) {  // rows cannot be attributed to trajectories
    if (a.sums_out && threadIdx.x == 0) a.sums_out[2 * i] = a.sums_out[2 * i + 1] = 0.0;
    return;
  }
  // the trajectory's rows in this call, as local indices [lo, hi)
  const long long lo = max(static_cast<long long>(a.cu[i]), a.row0) - a.row0;
  const long long hi = max(min(static_cast<long long>(a.cu[i + 1]), a.row0 + a.R) - a.row0, lo);
  const int n_i = ws.traj_n[i];
  const LossScalars& s = a.s;

  // sums over the trajectory's training tokens: log-ratio and correction weight
  double sl = 0.0, sw = 0.0;
  if (!a.sums_in) {
    for (long long t = lo + threadIdx.x; t < hi; t += kThreads) {
      if (!a.mask[t]) continue;
      const float base = a.old ? a.old[t] : a.rho[t];
      sl += static_cast<double>(ws.logp[t]) - static_cast<double>(base);
      sw += correction_weight(ws.rc[t], s);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    sl += __shfl_xor_sync(0xffffffffu, sl, o);
    sw += __shfl_xor_sync(0xffffffffu, sw, o);
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) { s_a[warp] = sl; s_b[warp] = sw; }
  __syncthreads();
  if (threadIdx.x == 0) {
    double tl = 0.0, tw = 0.0;
    for (int w = 0; w < kWarps; ++w) { tl += s_a[w]; tw += s_b[w]; }
    if (a.sums_in) {
      tl = a.sums_in[2 * i];
      tw = a.sums_in[2 * i + 1];
    }
    if (a.sums_out) {
      a.sums_out[2 * i] = tl;
      a.sums_out[2 * i + 1] = tw;
    }
    float si = 1.0f, pg = 0.0f, gp = 0.0f;
    uint8_t fl = 0;
    if (n_i > 0) {
      si = static_cast<float>(exp(tl / n_i));
      const float A = ws.a_traj[i];
      const float u = -A * si;
      const float c = -A * fminf(fmaxf(si, 1.0f - s.eps_lo), 1.0f + s.eps_hi);
      const bool clipped = c > u;
      pg = clipped ? c : u;
      if (clipped && si > 1.0f + s.eps_hi) fl |= kFlagClipHi;
      if (clipped && si < 1.0f - s.eps_lo) fl |= kFlagClipLo;
      bool dual = false;
      if (s.dual_c > 0.0f && A < 0.0f) {
        const float d = -A * s.dual_c;
        if (d < pg) { pg = d; dual = true; fl |= kFlagDual; }
      }
      const double n_seq = static_cast<double>(ws.hdr->n_seq);
      const double N = static_cast<double>(ws.hdr->n_tokens);
      const float scale = static_cast<float>(N / (n_seq * n_i));
      pg *= scale;
      gp = (clipped || dual) ? 0.0f : scale * static_cast<float>(tw / n_i) * (-A * si);
    }
    s_out[0] = si;
    s_out[1] = pg;
    s_out[2] = gp;
    s_out[3] = static_cast<float>(fl);
  }
  __syncthreads();
  if (a.sums_out) return;  // the shard's part of the sums only
  const float si = s_out[0], pg_i = s_out[1], gp = s_out[2];
  const uint8_t seq_flags = static_cast<uint8_t>(s_out[3]);
  for (long long t = lo + threadIdx.x; t < hi; t += kThreads) {
    const uint8_t keep = ws.flags[t] & (kFlagCorrClip | kFlagBad);
    if (keep & kFlagBad) continue;  // a row with a bad target keeps its zeros
    const float wt = correction_weight(ws.rc[t], s);
    float gkl = 0.0f;
    if (a.q) gkl = -expm1f(a.q[t] - ws.logp[t]);
    const float pg = n_i > 0 ? pg_i * wt : 0.0f;
    ws.r[t] = si;
    ws.pg[t] = pg;
    ws.ell[t] = pg + s.beta * ws.k3[t] - s.gamma * ws.H[t];
    ws.G[t] = gp + s.beta * gkl;
    ws.flags[t] = keep | seq_flags;
  }
}

}  // namespace

const void* seq_kernel() { return reinterpret_cast<const void*>(&k_seq); }

}  // namespace milesloss

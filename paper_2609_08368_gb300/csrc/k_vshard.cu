// The merge step of a vocabulary-sharded call (tensor parallelism: each rank
// holds a block of the vocabulary's columns, as in the paper's case study,
// Sec. 9.1, TP 2). The forward sweep of every shard wrote one record of two
// float4 per row over its own columns:
//   first   m   a reference in log2 units (a multiple of k = log2(e) / T of
//               a logit),
//           s   sum_j 2^(z_j k - m),
//           u   sum_j 2^(z_j k - m) (z_j k - m),
//           zy  the target's logit when the target is one of the shard's
//               columns, else 0;
//           m = NaN marks a row that shard gave up on (a timed-out wait);
//   second  with top-K OPD (Sec. 5.2), the part of the row's candidates in
//           the shard's columns: mt = the largest z_c k, sw = sum_c
//           2^(z_c k - mt), acc = sum_c 2^(z_c k - mt) (z_c / T - teacher_c),
//           and 1 when a candidate id lies outside the vocabulary (else 0);
//           (-inf, 0, 0, 0) without candidates there.
// The caller gathers the records of all shards (shard-major: the record of
// shard k and row r at all[2 (k R + r)]); here each row's records are merged
// in shard order, which gives every shard the same bits, and the row's
// statistics, log-prob, entropy and per-token objective are written as the
// fused sweep's epilogue writes them:
//   lse = M ln 2 + ln S,  H = ln S - U ln 2 / S,  logp = z_y / T - lse,
//   top-K signal = ACC / SW - lse (A -= opd_coef times it)
// (Sec. 3.4 ratio and the objective in token_terms). The gradient sweep
// (k_bwd over the shard's columns) and the statistics then read them.
#include "common.cuh"
#include "kernels.h"

namespace milesloss {

namespace {

constexpr float kLn2f = 0.69314718055994531f;

__global__ void __launch_bounds__(kMergeThreads) k_vmerge(const MergeArgs a) {
  WsPtrs ws = a.ws;
  uint32_t* err = &ws.hdr->err_bits;
  const long long V_total = a.col_starts[a.n_shards];
  for (long long row = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; row < a.R;
       row += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long y = a.targets[row];
    const bool yok = y >= 0 && y < V_total;
    // the shard whose columns hold the target
    int owner = -1;
    if (yok)
      for (int k = 0; k < a.n_shards; ++k)
        if (y >= a.col_starts[k] && y < a.col_starts[k + 1]) owner = k;
    const bool topk = a.s.topk > 0;
    float M = -INFINITY, Mt = -INFINITY, zy = 0.0f;
    bool gave_up = false, tk_bad = false;
    for (int k = 0; k < a.n_shards; ++k) {
      const long long at = 2 * (k * a.R + row);
      const float4 e = a.all[at];
      if (isnan(e.x)) gave_up = true;
      else if (e.y > 0.0f) M = fmaxf(M, e.x);
      if (k == owner) zy = e.w;
      if (topk) {
        const float4 c = a.all[at + 1];
        if (c.y > 0.0f) Mt = fmaxf(Mt, c.x);
        if (c.w != 0.0f) tk_bad = true;
      }
    }
    float S = 0.0f, U = 0.0f, SW = 0.0f, ACC = 0.0f;
    for (int k = 0; k < a.n_shards; ++k) {
      const long long at = 2 * (k * a.R + row);
      const float4 e = a.all[at];
      if (e.y > 0.0f) {  // (false for a NaN-marked record)
        const float d = e.x - M, f = ex2(d);
        S += f * e.y;
        U += f * fmaf(d, e.y, e.z);
      }
      if (topk) {
        const float4 c = a.all[at + 1];
        if (c.y > 0.0f) {
          const float f = ex2(c.x - Mt);
          SW = fmaf(f, c.y, SW);
          ACC = fmaf(f, c.z, ACC);
        }
      }
    }
    if (!yok) atomicOr(err, kErrTarget);
    if (tk_bad) atomicOr(err, kErrTopK);
    const bool bad = !yok || gave_up || tk_bad;
    const float lnS = logf(S);
    const float lse = fmaf(M, kLn2f, lnS);
    float H = lnS - U * kLn2f / S;
    float logp = zy * a.s.invT - lse;
    if (bad) { logp = 0.0f; H = 0.0f; }
    const float rho = a.rho[row];
    const float q = a.q ? a.q[row] : 0.0f;
    const float old = a.old ? a.old[row] : 0.0f;
    float A = ws.a_row[row];
    // top-K OPD signal (Sec. 5.2), a fixed per-token reward (SW >= 1 when
    // the row has a candidate)
    if (topk && !bad && SW > 0.0f) A -= a.s.opd_coef * (__fdividef(ACC, SW) - lse);
    TokenTerms tt = token_terms(logp, H, rho, q, a.q != nullptr, old, a.old != nullptr, A, a.s);
    if (bad) tt = TokenTerms{0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, kFlagBad};
    if (a.out_logp) a.out_logp[row] = logp;
    if (a.out_H) a.out_H[row] = H;
    ws.logp[row] = logp;
    ws.H[row] = H;
    ws.lse[row] = lse;
    ws.G[row] = tt.G;
    ws.ell[row] = tt.ell;
    ws.pg[row] = tt.pg;
    ws.k3[row] = tt.k3;
    ws.r[row] = tt.r;
    ws.rc[row] = tt.rc;
    ws.flags[row] = tt.flags;
  }
}

}  // namespace

const void* merge_kernel() { return reinterpret_cast<const void*>(&k_vmerge); }

}  // namespace milesloss

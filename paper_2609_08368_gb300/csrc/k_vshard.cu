// The merge step of a vocabulary-sharded call (tensor parallelism: each rank
// holds a block of the vocabulary's columns, as in the paper's case study,
// Sec. 9.1, TP 2). The forward sweep of every shard wrote one record per row
// over its own columns (a float4):
//   m   a reference in log2 units (a multiple of k = log2(e) / T of a logit),
//   s   sum_j 2^(z_j k - m),
//   u   sum_j 2^(z_j k - m) (z_j k - m),
//   zy  the target's logit when the target is one of the shard's columns,
//       else 0;
// m = NaN marks a row that shard gave up on (a timed-out wait). The caller
// gathers the records of all shards (shard-major: all[k * R + row]); here
// each row's records are merged in shard order, which gives every shard the
// same bits, and the row's statistics, log-prob, entropy and per-token
// objective are written as the fused sweep's epilogue writes them:
//   lse = M ln 2 + ln S,  H = ln S - U ln 2 / S,  logp = z_y / T - lse
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
    float M = -INFINITY, zy = 0.0f;
    bool gave_up = false;
    for (int k = 0; k < a.n_shards; ++k) {
      const float4 e = a.all[k * a.R + row];
      if (isnan(e.x)) gave_up = true;
      else if (e.y > 0.0f) M = fmaxf(M, e.x);
      if (k == owner) zy = e.w;
    }
    float S = 0.0f, U = 0.0f;
    for (int k = 0; k < a.n_shards; ++k) {
      const float4 e = a.all[k * a.R + row];
      if (e.y > 0.0f) {  // (false for a NaN-marked record)
        const float d = e.x - M, f = ex2(d);
        S += f * e.y;
        U += f * fmaf(d, e.y, e.z);
      }
    }
    if (!yok) atomicOr(err, kErrTarget);
    const bool bad = !yok || gave_up;
    const float lnS = logf(S);
    const float lse = fmaf(M, kLn2f, lnS);
    float H = lnS - U * kLn2f / S;
    float logp = zy * a.s.invT - lse;
    if (bad) { logp = 0.0f; H = 0.0f; }
    const float rho = a.rho[row];
    const float q = a.q ? a.q[row] : 0.0f;
    const float old = a.old ? a.old[row] : 0.0f;
    TokenTerms tt = token_terms(logp, H, rho, q, a.q != nullptr, old, a.old != nullptr,
                                ws.a_row[row], a.s);
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

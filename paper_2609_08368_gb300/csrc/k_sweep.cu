// The vocabulary sweep: per row, the tempered log-softmax statistics, the
// sampled token's log-prob, the entropy, the per-token objective and (when
// kGrad) dLogits, reading each logit from HBM exactly once.
//
// Layout of the work. A thread-block cluster of C CTAs owns one row at a
// time; CTA c of the cluster owns the columns [c*slice, c*slice + slice) of
// every row the cluster visits (rows cluster_id, cluster_id + n_clusters,
// ...). Each CTA streams its slices into an S-stage shared-memory ring with
// bulk async copies (cp.async.bulk, completion counted on an mbarrier per
// stage), so the copies of the next S-1 rows are in flight while the current
// one is processed. Per row:
//   pass A  every thread folds its elements into an online (max m, sum S of
//           2^(t - m k), sum U of 2^(t - m k) (t - m k)) with t = z log2(e)/T;
//           warp shuffles, then one warp, combine the threads in a fixed
//           order; CTAs exchange their triples through distributed shared
//           memory and every CTA combines the C triples in rank order, so all
//           CTAs of the cluster hold bit-identical row statistics;
//   epilogue one thread evaluates the per-token objective (ratio, clips, k3,
//           entropy term) and the coefficients of the gradient;
//   pass B  (kGrad) the slice is swept again from shared memory and dLogits
//           is written with 16-byte streaming stores.
// Definitions: Sec. 3.4 (ratio), Sec. 2 / 9.1 (group-relative advantage),
// Sec. 2.4 (loss mask); the gradient is the chain rule through them.
#include "common.cuh"
#include "kernels.h"

namespace milesloss {

namespace {

constexpr int kThreads = kSweepThreads;
constexpr int kWarps = kThreads / 32;
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s per bulk-copy wait
constexpr float kLn2 = 0.69314718055994531f;

struct Tri {
  float m, s, u;  // max of z; sum of 2^(t - m k); sum of 2^(t - m k) (t - m k)
};

// Merge two triples (k = log2(e)/T). Commutative bit-for-bit, so butterfly
// reductions leave every lane with the same value.
__device__ __forceinline__ Tri merge(Tri a, Tri b, float k) {
  if (b.s == 0.0f) return a;
  if (a.s == 0.0f) return b;
  const float m = fmaxf(a.m, b.m);
  const float da = (a.m - m) * k, db = (b.m - m) * k;
  const float fa = ex2(da), fb = ex2(db);
  Tri r;
  r.m = m;
  r.s = fa * a.s + fb * b.s;
  r.u = fa * fmaf(da, a.s, a.u) + fb * fmaf(db, b.s, b.u);
  return r;
}

__device__ __forceinline__ Tri shfl_xor(Tri t, int o) {
  Tri r;
  r.m = __shfl_xor_sync(0xffffffffu, t.m, o);
  r.s = __shfl_xor_sync(0xffffffffu, t.s, o);
  r.u = __shfl_xor_sync(0xffffffffu, t.u, o);
  return r;
}

__device__ __forceinline__ Tri warp_merge(Tri t, float k) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t = merge(t, shfl_xor(t, o), k);
  return t;
}

// Block-wide merge; the result is valid in warp 0. Contains a __syncthreads.
__device__ __forceinline__ Tri block_merge(Tri t, float k, float4* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  t = warp_merge(t, k);
  if (lane == 0) red[warp] = make_float4(t.m, t.s, t.u, 0.0f);
  __syncthreads();
  if (warp == 0) {
    Tri x{-INFINITY, 0.0f, 0.0f};
    if (lane < kWarps) {
      const float4 v = red[lane];
      x = Tri{v.x, v.y, v.z};
    }
    t = warp_merge(x, k);
  }
  return t;
}

// Fold one value into a thread's running triple (two interleaved sums).
struct Acc {
  float m = -INFINITY, mt = -INFINITY, s0 = 0.0f, s1 = 0.0f, u0 = 0.0f, u1 = 0.0f;

  __device__ __forceinline__ void raise(float vm, float k) {
    if (vm > m) {
      if (s0 + s1 > 0.0f) {
        const float d = (m - vm) * k, f = ex2(d);
        u0 = f * fmaf(d, s0, u0);
        u1 = f * fmaf(d, s1, u1);
        s0 *= f;
        s1 *= f;
      }
      m = vm;
      mt = vm * k;
    }
  }
  // t below -127 contributes 0 either way; the clamp keeps -inf logits
  // from producing 0 * -inf.
  __device__ __forceinline__ void add0(float z, float k) {
    const float t = fmaxf(fmaf(z, k, -mt), -127.0f);
    const float x = ex2(t);
    s0 += x;
    u0 = fmaf(x, t, u0);
  }
  __device__ __forceinline__ void add1(float z, float k) {
    const float t = fmaxf(fmaf(z, k, -mt), -127.0f);
    const float x = ex2(t);
    s1 += x;
    u1 = fmaf(x, t, u1);
  }
  __device__ __forceinline__ Tri tri() const { return Tri{m, s0 + s1, u0 + u1}; }
};

template <class In, class Out, bool kGrad>
__global__ void __launch_bounds__(kThreads, 1) k_sweep(const SweepArgs a) {
  using St = typename In::storage;
  constexpr int V8 = In::kVec;
  extern __shared__ __align__(128) unsigned char smem[];
  const int tid = threadIdx.x;
  const int C = static_cast<int>(cluster_nctarank());
  const int crank = static_cast<int>(cluster_ctarank());
  const long long cl_id = blockIdx.x / C;
  const long long n_cl = gridDim.x / C;
  const int S = a.stages;
  const int slice = a.slice;
  const int lo = crank * slice;
  const int cnt = max(0, min(slice, a.V - lo));
  const int n_vec = a.in_bulk ? cnt / V8 : 0;
  const int vec_elems = n_vec * V8;
  const uint32_t bulk_bytes = static_cast<uint32_t>(n_vec) * 16u;
  const float k = a.s.k;

  unsigned char* stages = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(S) * a.stage_bytes);
  float4* xch = reinterpret_cast<float4*>(bars + kMaxStages);  // [2]
  float4* red = xch + 2;                                        // [kWarps]
  float4* bc = red + kWarps;                                    // [1]
  int4* bci = reinterpret_cast<int4*>(bc + 1);                  // [1]

  WsPtrs ws = a.ws;
  const long long N = ws.hdr->n_tokens;
  float g = a.grad_loss;
  if (a.grad_loss_dev) g *= *a.grad_loss_dev;
  const float cscale = (N > 0) ? g / static_cast<float>(N) * a.s.invT : 0.0f;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) mbar_init(smem_u32(&bars[s]), 1);
    fence_mbar_init();
  }
  __syncthreads();

  const uint64_t pol = l2_policy_evict_first();
  const char* lg = static_cast<const char*>(a.logits);
  auto row_src = [&](long long row) -> const char* {
    return lg + (row * a.ld + lo) * static_cast<long long>(sizeof(St));
  };
  // Bit s of iss_par is the phase parity of the next copy into stage s.
  uint32_t iss_par = 0, iss_any = 0;
  auto issue = [&](int s, long long row) {
    iss_par ^= 1u << s;
    iss_any |= 1u << s;
    const uint32_t bar = smem_u32(&bars[s]);
    const uint32_t dst = smem_u32(stages + static_cast<size_t>(s) * a.stage_bytes);
    const char* src = row_src(row);
    mbar_arrive_expect_tx(bar, bulk_bytes);
    for (uint32_t off = 0; off < bulk_bytes; off += kBulkChunk) {
      const uint32_t n = min(kBulkChunk, bulk_bytes - off);
      bulk_g2s(dst + off, src + off, n, bar, pol);
    }
  };

  bool dead = false;
  if (tid == 0 && bulk_bytes) {
    for (int s = 0; s < S; ++s) {
      const long long row = cl_id + s * n_cl;
      if (row < a.R) issue(s, row);
    }
  }

  long long it = 0;
  for (long long row = cl_id; row < a.R; row += n_cl, ++it) {
    const int s = static_cast<int>(it % S);
    const uint32_t parity = static_cast<uint32_t>((it / S) & 1);
    const unsigned char* sb = stages + static_cast<size_t>(s) * a.stage_bytes;
    const char* grow = row_src(row);

    // Row scalars for the epilogue; their latency hides behind pass A.
    int y = 0;
    float rho = 0.0f, q = 0.0f, old = 0.0f, A = 0.0f;
    uint8_t msk = 0;
    if (tid == 0) {
      y = a.targets[row];
      rho = a.rho[row];
      if (a.q) q = a.q[row];
      if (a.old) old = a.old[row];
      A = ws.a_row[row];
      msk = a.mask[row];
    }

    if (bulk_bytes && !dead) {
      if (!mbar_wait_bounded(smem_u32(&bars[s]), parity, kWaitLimitNs)) {
        dead = true;
        atomicOr(&ws.hdr->err_bits, kErrTimeout);
      }
    }

    // ---------------- pass A
    Acc acc;
    const uint4* sv = reinterpret_cast<const uint4*>(sb);
#pragma unroll 2
    for (int v = tid; v < n_vec; v += kThreads) {
      const uint4 w = sv[v];
      acc.raise(In::vmax(w), k);
      float f[V8];
      In::unpack(w, f);
#pragma unroll
      for (int e = 0; e < V8; e += 2) {
        acc.add0(f[e], k);
        acc.add1(f[e + 1], k);
      }
    }
    for (int j = vec_elems + tid; j < cnt; j += kThreads) {
      const float z = In::load1(grow, j);
      acc.raise(z, k);
      acc.add0(z, k);
    }
    Tri t = block_merge(acc.tri(), k, red);

    // ---------------- cluster exchange and epilogue
    const bool yok = (tid == 0) && (y >= 0) && (y < a.V);
    const int owner = yok ? y / slice : -1;
    if (tid == 0) {
      float zy = 0.0f;
      if (owner == crank) {
        const int jl = y - lo;
        zy = (jl < vec_elems) ? In::load1(sb, jl) : In::load1(grow, jl);
      }
      xch[it & 1] = make_float4(t.m, t.s, t.u, zy);
    }
    if (C > 1) {
      cluster_sync_all();
    } else {
      __syncthreads();
    }
    if (tid == 0) {
      Tri tot{-INFINITY, 0.0f, 0.0f};
      float zy = 0.0f;
      const uint32_t mine = smem_u32(&xch[it & 1]);
      for (int r = 0; r < C; ++r) {
        const float4 e = (C > 1) ? ld_dsmem_f4(mapa_shared(mine, r)) : xch[it & 1];
        tot = merge(tot, Tri{e.x, e.y, e.z}, k);
        if (r == owner) zy = e.w;
      }
      const bool bad = !yok;
      if (bad) atomicOr(&ws.hdr->err_bits, kErrTarget);
      const float lnS = logf(tot.s);
      const float lse = tot.m * a.s.invT + lnS;
      float H = lnS - tot.u * kLn2 / tot.s;
      float logp = zy * a.s.invT - lse;
      if (bad) { logp = 0.0f; H = 0.0f; }
      TokenTerms tt = token_terms(logp, H, rho, q, a.q != nullptr, old, a.old != nullptr, A, a.s);
      if (bad) tt = TokenTerms{0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, kFlagBad};
      if (crank == 0) {
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
      if (kGrad) {
        // dZ_j = p_j (ca + cb z_j) + add 1[j = y],  p_j = 2^(z_j k - L2)
        const float cc = (msk && !bad) ? cscale : 0.0f;
        const float ca = cc * (-tt.G + a.s.gamma * (H - lse));
        const float cb = cc * a.s.gamma * a.s.invT;
        const float add = cc * tt.G;
        const float L2 = tot.m * k + __log2f(tot.s);
        const bool zero = (cc == 0.0f) || (ca == 0.0f && cb == 0.0f);
        const bool fold = !zero && (cb == 0.0f);
        // fold: p_j ca = sign(ca) 2^(z_j k - L2 + log2|ca|)
        const float off = fold ? (__log2f(fabsf(ca)) - L2) : -L2;
        bc[0] = make_float4(off, ca, cb, add);
        bci[0] = make_int4(zero, fold, (fold && ca < 0.0f) ? 1 : 0,
                           (owner == crank && !zero) ? y - lo : -1);
      }
    }
    __syncthreads();

    // ---------------- pass B
    if (kGrad) {
      const float4 c = bc[0];
      const int4 ci = bci[0];
      char* drow = static_cast<char*>(a.dlogits) +
                   (row * a.ld_out + lo) * static_cast<long long>(Out::kSize);
      const int nvo = a.out_vec ? n_vec : 0;
      const int vo_elems = nvo * V8;
      if (ci.x) {
        float zf[V8];
#pragma unroll
        for (int e = 0; e < V8; ++e) zf[e] = 0.0f;
        for (int v = tid; v < nvo; v += kThreads)
          Out::template storev<V8>(drow + static_cast<size_t>(v) * V8 * Out::kSize, zf, 0u);
        for (int j = vo_elems + tid; j < cnt; j += kThreads) Out::store1(drow, j, 0.0f);
      } else if (ci.y) {
        const uint32_t sgn = ci.z ? Out::kSignMask : 0u;
#pragma unroll 2
        for (int v = tid; v < nvo; v += kThreads) {
          float f[V8];
          In::unpack(sv[v], f);
#pragma unroll
          for (int e = 0; e < V8; ++e) f[e] = ex2(fmaf(f[e], k, c.x));
          Out::template storev<V8>(drow + static_cast<size_t>(v) * V8 * Out::kSize, f, sgn);
        }
        for (int j = vo_elems + tid; j < cnt; j += kThreads) {
          const float z = (j < vec_elems) ? In::load1(sb, j) : In::load1(grow, j);
          const float x = ex2(fmaf(z, k, c.x));
          Out::store1(drow, j, ci.z ? -x : x);
        }
      } else {
#pragma unroll 2
        for (int v = tid; v < nvo; v += kThreads) {
          float f[V8];
          In::unpack(sv[v], f);
#pragma unroll
          for (int e = 0; e < V8; ++e) f[e] = ex2(fmaf(f[e], k, c.x)) * fmaf(c.z, f[e], c.y);
          Out::template storev<V8>(drow + static_cast<size_t>(v) * V8 * Out::kSize, f, 0u);
        }
        for (int j = vo_elems + tid; j < cnt; j += kThreads) {
          const float z = (j < vec_elems) ? In::load1(sb, j) : In::load1(grow, j);
          Out::store1(drow, j, ex2(fmaf(z, k, c.x)) * fmaf(c.z, z, c.y));
        }
      }
      __syncthreads();
      if (tid == 0 && ci.w >= 0) {
        // the sampled token's entry gets + cc G (the one-hot term)
        const int jl = ci.w;
        const float z = (jl < vec_elems) ? In::load1(sb, jl) : In::load1(grow, jl);
        float x;
        if (ci.y) {
          x = ex2(fmaf(z, k, c.x));
          if (ci.z) x = -x;
        } else {
          x = ex2(fmaf(z, k, c.x)) * fmaf(c.z, z, c.y);
        }
        Out::store1(drow, jl, x + c.w);
      }
    }

    // Refill this stage with the row S iterations ahead.
    if (tid == 0 && bulk_bytes && !dead) {
      const long long nrow = row + S * n_cl;
      if (nrow < a.R) {
        fence_proxy_async_smem();
        issue(s, nrow);
      }
    }
  }

  // Copies issued but never waited on exist only after a timeout: wait
  // (bounded) for the last copy into every stage before leaving.
  if (dead && tid == 0) {
    for (int s = 0; s < S; ++s)
      if (iss_any & (1u << s))
        mbar_wait_bounded(smem_u32(&bars[s]), ((iss_par >> s) & 1u) ^ 1u, kWaitLimitNs);
  }
  // No CTA may leave while a peer can still read its exchange slot.
  if (C > 1) cluster_sync_all();
}

}  // namespace

template <class In, class Out, bool kGrad>
static const void* sweep_fn() {
  return reinterpret_cast<const void*>(&k_sweep<In, Out, kGrad>);
}

const void* sweep_kernel(rl_dtype in, rl_dtype out, bool grad) {
  if (!grad) return in == RL_BF16 ? sweep_fn<InBf16, OutBf16, false>()
                                  : sweep_fn<InF32, OutF32, false>();
  if (in == RL_BF16) return out == RL_BF16 ? sweep_fn<InBf16, OutBf16, true>()
                                           : sweep_fn<InBf16, OutF32, true>();
  return out == RL_BF16 ? sweep_fn<InF32, OutBf16, true>() : sweep_fn<InF32, OutF32, true>();
}

}  // namespace milesloss

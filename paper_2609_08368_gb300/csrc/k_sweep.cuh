// The vocabulary sweep: per row, the tempered log-softmax statistics, the
// sampled token's log-prob, the entropy, the per-token objective and (when
// kGrad) dLogits, reading each logit from HBM exactly once.
//
// Layout of the work. A thread-block cluster of C CTAs owns one row at a
// time; CTA c of the cluster owns the columns [c*slice, c*slice + slice) of
// every row the cluster visits (rows cluster_id, cluster_id + n_clusters,
// ...). Each CTA streams its slices into an S-stage shared-memory ring with
// bulk async copies (cp.async.bulk, completion counted on an mbarrier per
// stage). Several CTAs share an SM, so one CTA's per-row synchronisation
// overlaps the others' arithmetic. Per row:
//   pass A  every thread sums S = sum 2^(t - r) and U = sum 2^(t - r) (t - r),
//           t = z log2(e)/T, two lanes per instruction (f32x2), against a
//           reference r taken from its first vector (a second sweep for the
//           maximum runs only on overflow or -inf logits); warp shuffles,
//           then one warp, merge the threads' (r, S, U) in a fixed order;
//   exchange thread 0 pushes the CTA's (m, S, U, z_y) into every peer's
//           shared memory with st.async, counted on the peer's mbarrier,
//           and merges the C triples in rank order once they have all
//           arrived, so every CTA of the cluster holds bit-identical row
//           statistics;
//   epilogue thread 0 evaluates the per-token objective and the gradient
//           coefficients;
//   pass B  (kGrad) the slice is swept again from shared memory and dLogits
//           is written with 16-byte streaming stores.
// Definitions: Sec. 3.4 (ratio), Sec. 2 / 9.1 (group-relative advantage),
// Sec. 2.4 (loss mask); the gradient is the chain rule through them.
#pragma once

#include <type_traits>

#include "common.cuh"
#include "kernels.h"

namespace milesloss {

namespace {

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s per bounded wait
constexpr float kLn2 = 0.69314718055994531f;

// Partial sums against a reference r in log2 units (t = z k, k = log2(e)/T):
// s = sum 2^(t - r), u = sum 2^(t - r) (t - r). Any finite r gives the same
// row statistics: lse = r ln 2 + ln s, H = ln s - u ln 2 / s.
struct Tri {
  float m, s, u;  // m = r
};

// Warp-wide merge in a fixed order: the largest reference first, then every
// lane rescales its sums once to it, then plain butterfly sums. Every lane
// ends with the same triple.
__device__ __forceinline__ Tri warp_merge(Tri t) {
  float M = t.m;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  float s = 0.0f, u = 0.0f;
  if (t.s > 0.0f) {
    const float d = t.m - M, f = ex2(d);
    s = f * t.s;
    u = f * fmaf(d, t.s, t.u);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    s += __shfl_xor_sync(0xffffffffu, s, o);
    u += __shfl_xor_sync(0xffffffffu, u, o);
  }
  return Tri{M, s, u};
}

// Block-wide merge; the result is valid in warp 0. Contains a __syncthreads.
template <int kWarps>
__device__ __forceinline__ Tri block_merge(Tri t, float4* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  t = warp_merge(t);
  if (lane == 0) red[warp] = make_float4(t.m, t.s, t.u, 0.0f);
  __syncthreads();
  if (warp == 0) {
    Tri x{-INFINITY, 0.0f, 0.0f};
    if (lane < kWarps) {
      const float4 v = red[lane];
      x = Tri{v.x, v.y, v.z};
    }
    t = warp_merge(x);
  }
  return t;
}

// Sum of 2^(t - mt) and of 2^(t - mt) (t - mt) over the thread's vectors,
// t = z k, for a fixed reference mt in log2 units. kSafe skips
// -inf logits exactly (0 * -inf would otherwise give NaN); it runs only
// when the fast pass produced a NaN.
template <class In, int kThreads, bool kSafe>
__device__ __forceinline__ void sum_pass(const uint4* sv, int n_vec, float k, float mt,
                                         float& s_out, float& u_out) {
  constexpr int P = In::kVec / 2;  // pairs per 16 bytes
  const float2 k2 = make_float2(k, k);
  const float2 nm2 = make_float2(-mt, -mt);
  float2 s0 = make_float2(0.0f, 0.0f), s1 = s0, u0 = s0, u1 = s0;
  int v = threadIdx.x;
  for (; v + kThreads < n_vec; v += 2 * kThreads) {
    float2 fa[P], fb[P];
    In::unpack2(sv[v], fa);
    In::unpack2(sv[v + kThreads], fb);
#pragma unroll
    for (int e = 0; e < P; ++e) {
      float2 ta = ffma2(fa[e], k2, nm2), tb = ffma2(fb[e], k2, nm2);
      if (kSafe) {
        if (fa[e].x == -INFINITY) ta.x = -127.0f;
        if (fa[e].y == -INFINITY) ta.y = -127.0f;
        if (fb[e].x == -INFINITY) tb.x = -127.0f;
        if (fb[e].y == -INFINITY) tb.y = -127.0f;
      }
      const float2 xa = ex2x2(ta), xb = ex2x2(tb);
      s0 = fadd2(s0, xa);
      s1 = fadd2(s1, xb);
      u0 = ffma2(xa, ta, u0);
      u1 = ffma2(xb, tb, u1);
    }
  }
  if (v < n_vec) {
    float2 fa[P];
    In::unpack2(sv[v], fa);
#pragma unroll
    for (int e = 0; e < P; ++e) {
      float2 ta = ffma2(fa[e], k2, nm2);
      if (kSafe) {
        if (fa[e].x == -INFINITY) ta.x = -127.0f;
        if (fa[e].y == -INFINITY) ta.y = -127.0f;
      }
      const float2 xa = ex2x2(ta);
      s0 = fadd2(s0, xa);
      u0 = ffma2(xa, ta, u0);
    }
  }
  const float2 s = fadd2(s0, s1), u = fadd2(u0, u1);
  s_out = s.x + s.y;
  u_out = u.x + u.y;
}

// The thread's sums against its own maximum over the slice, skipping -inf
// logits exactly: the rare path (no finite first vector, an overflow, or a
// -inf logit).
template <class In, int kThreads>
__device__ __forceinline__ Tri slow_sums(const uint4* sv, int n_vec, float k) {
  typename In::MaxAcc macc = In::kMaxInit;
  for (int v = threadIdx.x; v < n_vec; v += kThreads) macc = In::max_acc(macc, sv[v]);
  const float r = In::max_val(macc) * k;
  Tri t{-INFINITY, 0.0f, 0.0f};
  if (r != -INFINITY) {
    float su, uu;
    sum_pass<In, kThreads, true>(sv, n_vec, k, r, su, uu);
    t = Tri{r, su, uu};
  }
  return t;
}

template <class In, class Out, bool kGrad, int kThreads, int kMinBlocks, bool kTopK>
__global__ void __launch_bounds__(kThreads, kMinBlocks) k_sweep(const SweepArgs a) {
  using St = typename In::storage;
  constexpr int V8 = In::kVec;
  constexpr int P = V8 / 2;
  constexpr int kWarps = kThreads / 32;
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
  uint64_t* xbar = bars + kMaxStages;                          // [2] exchange barriers
  // [2][2 kMaxCluster]: per slot, the CTAs' (m, S, U, z_y), then their top-K parts
  float4* xch = reinterpret_cast<float4*>(xbar + 2);
  float4* red = xch + 4 * kMaxCluster;                         // [kWarps]
  float4* bc = red + kWarps;                                   // [2]
  int4* bci = reinterpret_cast<int4*>(bc + 2);                 // [1]
  uint64_t* never = reinterpret_cast<uint64_t*>(bci + 1);      // [1] completed by nothing (test hook)
  volatile int* abort = reinterpret_cast<volatile int*>(never + 1);  // the CTA gave up
  static_assert(kMaxStages * 8 + 2 * 8 + 4 * kMaxCluster * 16 + (512 / 32 + 3) * 16 + 8 + 16 <=
                    kSweepSmemExtra,
                "k_sweep scratch");
  // [2] top-K candidates of this row and the next (launched with kTopKSmem more)
  TopKBuf* tkb = reinterpret_cast<TopKBuf*>(smem + static_cast<size_t>(S) * a.stage_bytes +
                                            kSweepSmemExtra);

  WsPtrs ws = a.ws;
  uint32_t* err = &ws.hdr->err_bits;
  const long long N = ws.hdr->n_tokens;
  float g = a.grad_loss;
  if (a.grad_loss_dev) g *= *a.grad_loss_dev;
  const float cscale = (N > 0) ? g / static_cast<float>(N) * a.s.invT : 0.0f;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) mbar_init(smem_u32(&bars[s]), 1);
    mbar_init(smem_u32(&xbar[0]), 1);
    mbar_init(smem_u32(&xbar[1]), 1);
    mbar_init(smem_u32(never), 1);
    *abort = 0;
    fence_mbar_init();
  }
  // Peers push into this CTA's exchange slots: all barriers must be
  // initialised cluster-wide first.
  if (C > 1) cluster_sync_all(); else __syncthreads();

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

  // Waits on the ring end early once any thread of the CTA has given up
  // (mbar_wait_or_abort); thread 0 then issues no more copies, and before
  // the CTA exits it waits (bounded) for the last copy into every stage, so
  // no bulk copy lands after the CTA is gone. The row exchange keeps its
  // own bounded waits (the peers' stores keep coming whatever this CTA
  // does); after one of them runs out, this CTA leaves the exchange
  // barriers alone.
  bool xdead = false;
  if (tid == 0 && bulk_bytes) {
    for (int s = 0; s < S; ++s) {
      const long long row = cl_id + s * n_cl;
      if (row < a.R) issue(s, row);
    }
  }

  constexpr bool topk = kTopK;  // top-K OPD on (a.s.topk > 0): its own instantiation
  if (topk && tid < 32 && cl_id < a.R)
    topk_prefetch(&tkb[0], a.s.topk_ids + cl_id * a.s.topk, a.s.topk_teacher + cl_id * a.s.topk,
                  a.s.topk, tid);

  long long it = 0;
  for (long long row = cl_id; row < a.R; row += n_cl, ++it) {
    const int s = static_cast<int>(it % S);
    const uint32_t parity = static_cast<uint32_t>((it / S) & 1);
    const unsigned char* sb = stages + static_cast<size_t>(s) * a.stage_bytes;
    const char* grow = row_src(row);
    const uint4* sv = reinterpret_cast<const uint4*>(sb);

    // Row scalars for the epilogue; their latency hides behind the passes.
    int y = 0;
    float rho = 0.0f, q = 0.0f, old = 0.0f, A = 0.0f;
    uint8_t msk = 0;
    if (tid == 0) {
      // the target's column in this call's logits (-1 outside them: a bad
      // target, or another shard's column in a vocabulary-sharded call)
      const long long yl = a.targets[row] - a.col0;
      y = (yl >= 0 && yl < a.V) ? static_cast<int>(yl) : -1;
      rho = a.rho[row];
      if (a.q) q = a.q[row];
      if (a.old) old = a.old[row];
      A = ws.a_row[row];
      msk = a.mask[row];
    }
    // top-K OPD candidates (warp 0): this row's ids and teacher values
    // arrived during the last row; the next row's are copied meanwhile
    const TopKBuf* tk_row = &tkb[it & 1];
    if (topk && tid < 32) {
      cp_async_wait_all();
      if (row + n_cl < a.R) {
        const long long o = (row + n_cl) * a.s.topk;
        topk_prefetch(&tkb[(it + 1) & 1], a.s.topk_ids + o, a.s.topk_teacher + o, a.s.topk, tid);
      }
    }

    bool have = true;  // the stage holds this row's slice (or nothing is copied)
    if (bulk_bytes) {
      if (it == 0 && a.stall_ns) {  // test hook: a barrier that nothing completes
        mbar_wait_or_abort(smem_u32(never), 0u, a.stall_ns, abort, err);
        have = false;
      } else {
        have = mbar_wait_or_abort(smem_u32(&bars[s]), parity, kWaitLimitNs, abort, err);
      }
    }

    // ---------------- pass A: one sweep against the maximum of the thread's
    // first vector. The sums stay finite unless a logit lies more than
    // 127 / k above that reference; that case (inf) or a -inf logit (NaN)
    // takes the thread's maximum over the slice and sums again, skipping
    // -inf logits exactly. Sums past 2^16 move the reference up by their
    // binary exponent (an exact rescale) before the merge.
    Tri t{-INFINITY, 0.0f, 0.0f};
    if (have && tid < n_vec) {
      const float r = In::vmax(sv[tid]) * k;
      if (r != -INFINITY) {
        float su, uu;
        sum_pass<In, kThreads, false>(sv, n_vec, k, r, su, uu);
        if (fabsf(su) < INFINITY && fabsf(uu) < INFINITY) t = Tri{r, su, uu};
      }
      if (t.m == -INFINITY) t = slow_sums<In, kThreads>(sv, n_vec, k);
      const int e = ((__float_as_int(t.s) >> 23) & 0xff) - 127;
      if (e > 16) {
        const float f = __int_as_float((127 - e) << 23), d = static_cast<float>(e);
        t.u = f * fmaf(-d, t.s, t.u);
        t.s *= f;
        t.m += d;
      }
    }
    for (int j = vec_elems + tid; j < cnt; j += kThreads) {  // elements past the vectors
      const float z = In::load1(grow, j);
      if (z == -INFINITY) continue;
      const float zk = z * k;
      if (zk > t.m) {
        if (t.s > 0.0f) {
          const float d = t.m - zk, f = ex2(d);
          t.u = f * fmaf(d, t.s, t.u);
          t.s *= f;
        }
        t.m = zk;
      }
      const float tt = fmaf(z, k, -t.m), x = ex2(tt);
      t.s += x;
      t.u = fmaf(x, tt, t.u);
    }
    // top-K OPD candidates in this CTA's columns (warp 0): from the slice in
    // shared memory, past its whole vectors from global memory
    TopKPart tkp{-INFINITY, 0.0f, 0.0f, 0};
    if (topk && tid < 32) {
      TopKLane tk = topk_ids(tk_row, static_cast<int>(a.col0), a.V, a.vocab_total, a.s.topk, tid);
      if (have) topk_gather<In>(tk, sb, lo, lo + vec_elems);
      topk_gather<In>(tk, grow + static_cast<size_t>(vec_elems) * sizeof(St), lo + vec_elems, lo + cnt);
      const int c0 = lo, c1 = lo + cnt;
      tkp = topk_part(tk, tk_row, tid, a.s.invT, k, [c0, c1](int id) { return id >= c0 && id < c1; });
    }
    t = block_merge<kWarps>(t, red);

    // ---------------- exchange and epilogue (thread 0)
    const bool yok = (tid == 0) && (y >= 0);
    const int owner = yok ? y / slice : -1;
    Tri tot{t.m, t.s, t.u};  // the row's statistics (thread 0)
    float zy_all = 0.0f;
    if (tid == 0) {
      float zy = 0.0f;
      if (owner == crank) {
        const int jl = y - lo;
        zy = (jl < vec_elems) ? (have ? In::load1(sb, jl) : 0.0f) : In::load1(grow, jl);
      }
      const int slot = static_cast<int>(it & 1);
      const float4 mine = make_float4(t.m, t.s, t.u, zy);
      const float4 mine_tk = make_float4(tkp.m, tkp.sw, tkp.acc, 0.0f);
      zy_all = zy;
      if (C > 1) {
        float4* xs = xch + slot * 2 * kMaxCluster;
        float4* xt = xs + kMaxCluster;
        xs[crank] = mine;
        xt[crank] = mine_tk;
        const uint32_t xaddr = smem_u32(&xs[crank]), taddr = smem_u32(&xt[crank]);
        const uint32_t xb = smem_u32(&xbar[slot]);
        for (int r = 0; r < C; ++r) {
          if (r == crank) continue;
          st_async_f4(mapa_shared(xaddr, r), mine, mapa_shared(xb, r));
          if (topk) st_async_f4(mapa_shared(taddr, r), mine_tk, mapa_shared(xb, r));
        }
        if (!xdead) {
          mbar_arrive_expect_tx(xb, static_cast<uint32_t>(C - 1) * (topk ? 32u : 16u));
          if (!mbar_wait_bounded(xb, static_cast<uint32_t>((it >> 1) & 1), kWaitLimitNs)) {
            xdead = true;
            *abort = 1;
            atomicOr(err, kErrTimeout);
          }
        }
        float M = -INFINITY;
        for (int r = 0; r < C; ++r) M = fmaxf(M, xs[r].x);
        tot = Tri{M, 0.0f, 0.0f};
        for (int r = 0; r < C; ++r) {
          const float4 e = xs[r];
          if (e.y > 0.0f) {
            const float d = e.x - M, f = ex2(d);
            tot.s += f * e.y;
            tot.u += f * fmaf(d, e.y, e.z);
          }
          if (r == owner) zy_all = e.w;
        }
        if (topk) {  // the CTAs' top-K parts (every CTA read the same ids)
          const int tk_bad = tkp.bad;
          tkp = topk_merge_all(xt, C);
          tkp.bad = tk_bad;
        }
      }
    }
    if (tid == 0 && a.part_rows) {
      // vocabulary-sharded forward: the row's partial sums over this
      // shard's columns (a row read after the CTA gave up is marked NaN)
      if (crank == 0) {
        a.part_rows[2 * row] = *abort ? make_float4(NAN, 0.0f, 0.0f, 0.0f)
                                      : make_float4(tot.m, tot.s, tot.u, yok ? zy_all : 0.0f);
        a.part_rows[2 * row + 1] = topk ? make_float4(tkp.m, tkp.sw, tkp.acc, tkp.bad ? 1.0f : 0.0f)
                                        : make_float4(-INFINITY, 0.0f, 0.0f, 0.0f);
      }
    } else if (tid == 0) {
      // a row read after the CTA gave up, a bad target or a bad top-K
      // candidate: zeros
      const bool bad = !yok || (topk && tkp.bad) || *abort;
      if (!yok && crank == 0) atomicOr(err, kErrTarget);
      if (topk && tkp.bad && crank == 0) atomicOr(err, kErrTopK);
      const float lnS = logf(tot.s);
      const float lse = fmaf(tot.m, kLn2, lnS);  // the reference is in log2 units
      float H = lnS - tot.u * kLn2 / tot.s;
      float logp = zy_all * a.s.invT - lse;
      if (bad) { logp = 0.0f; H = 0.0f; }
      // top-K OPD signal (Sec. 5.2), a fixed per-token reward
      if (topk && !bad) A -= a.s.opd_coef * topk_value(tkp, lse);
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
        // dZ_j = p_j (ca + cb z_j) + cc G 1[j = y],  p_j = 2^(z_j k - L2)
        const float cc = (msk && !bad) ? cscale : 0.0f;
        const float ca = cc * (-tt.G + a.s.gamma * (H - lse));
        const float cb = cc * a.s.gamma * a.s.invT;
        const float L2 = tot.m + __log2f(tot.s);
        const bool zero = (cc == 0.0f) || (ca == 0.0f && cb == 0.0f);
        const bool fold = !zero && (cb == 0.0f);
        // fold: p_j ca = sign(ca) 2^(z_j k - L2 + log2|ca|)
        const float off = fold ? (__log2f(fabsf(ca)) - L2) : -L2;
        bc[0] = make_float4(off, ca, cb, 0.0f);
        bc[1] = make_float4(logp, H, cc, tt.G);
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
      const float2 k2 = make_float2(k, k);
      const float2 off2 = make_float2(c.x, c.x);
      if (ci.x) {
        float zf[V8];
#pragma unroll
        for (int e = 0; e < V8; ++e) zf[e] = 0.0f;
        for (int v = tid; v < nvo; v += kThreads)
          Out::template storev<V8>(drow + static_cast<size_t>(v) * V8 * Out::kSize, zf, 0u);
        for (int j = vo_elems + tid; j < cnt; j += kThreads) Out::store1(drow, j, 0.0f);
      } else if (ci.y) {
        // p_j ca with |ca| folded into the exponent; the sign is applied
        // when packing (a negated operand costs no instruction).
        auto fold_loop = [&](auto neg) {
          constexpr bool kNeg = decltype(neg)::value;
#pragma unroll 2
          for (int v = tid; v < nvo; v += kThreads) {
            float2 f[P];
            In::unpack2(sv[v], f);
#pragma unroll
            for (int e = 0; e < P; ++e) {
              f[e] = ex2x2(ffma2(f[e], k2, off2));
              if (kNeg) f[e] = make_float2(-f[e].x, -f[e].y);
            }
            Out::template storev<V8>(drow + static_cast<size_t>(v) * V8 * Out::kSize,
                                     reinterpret_cast<const float*>(f), 0u);
          }
        };
        if (ci.z) fold_loop(std::true_type{}); else fold_loop(std::false_type{});
        for (int j = vo_elems + tid; j < cnt; j += kThreads) {
          const float z = (j < vec_elems) ? In::load1(sb, j) : In::load1(grow, j);
          const float x = ex2(fmaf(z, k, c.x));
          Out::store1(drow, j, ci.z ? -x : x);
        }
      } else {
        const float2 ca2 = make_float2(c.y, c.y), cb2 = make_float2(c.z, c.z);
#pragma unroll 2
        for (int v = tid; v < nvo; v += kThreads) {
          float2 f[P];
          In::unpack2(sv[v], f);
#pragma unroll
          for (int e = 0; e < P; ++e)
            f[e] = fmul2(ex2x2(ffma2(f[e], k2, off2)), ent_factor2(f[e], ca2, cb2));
          Out::template storev<V8>(drow + static_cast<size_t>(v) * V8 * Out::kSize,
                                   reinterpret_cast<const float*>(f), 0u);
        }
        for (int j = vo_elems + tid; j < cnt; j += kThreads) {
          const float z = (j < vec_elems) ? In::load1(sb, j) : In::load1(grow, j);
          Out::store1(drow, j, ex2(fmaf(z, k, c.x)) * ent_factor(z, c.y, c.z));
        }
      }
      __syncthreads();
      if (tid == 0 && ci.w >= 0) {
        // The sampled token's entry: cc [G (1 - p_y) + gamma p_y (log p_y + H)],
        // with 1 - p_y = -expm1(logp) so that p_y close to 1 keeps its
        // relative accuracy.
        const float4 ex = bc[1];  // logp, H, cc, G
        const float py = expf(ex.x);
        const float x = ex.z * (ex.w * -expm1f(ex.x) + a.s.gamma * py * (ex.x + ex.y));
        Out::store1(drow, ci.w, x);
      }
    }

    // Refill this stage with the row S iterations ahead.
    if (tid == 0 && bulk_bytes && !*abort) {
      const long long nrow = row + S * n_cl;
      if (nrow < a.R) {
        fence_proxy_async_smem();
        issue(s, nrow);
      }
    }
  }

  // Wait (bounded) for the last copy into every stage before leaving: at
  // once unless the CTA gave up with copies in flight.
  if (tid == 0) {
    for (int s = 0; s < S; ++s)
      if ((iss_any & (1u << s)) &&
          !mbar_wait_bounded(smem_u32(&bars[s]), ((iss_par >> s) & 1u) ^ 1u, kWaitLimitNs))
        atomicOr(err, kErrTimeout);
  }
  // No CTA leaves while a peer's last exchange store into it may be in flight.
  if (C > 1) cluster_sync_all();
}

}  // namespace

}  // namespace milesloss

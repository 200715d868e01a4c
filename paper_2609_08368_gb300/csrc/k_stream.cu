// The streaming vocabulary sweep, one CTA per row: the same per-row results
// as k_sweep (log-softmax statistics, log-prob, entropy, per-token
// objective, dLogits), with no exchange between CTAs (except in the cluster
// instantiation for the longest rows, below). Long rows run one CTA
// per SM with sixteen consumer warps; shorter rows two or four CTAs per SM
// with eight or four consumer warps each, so that one CTA's per-row merge and
// epilogue overlap the others' passes. Rows of 480 KB and more (fused calls
// without top-K) run on a cluster of two or four CTAs per row, each streaming
// a slice, so that fewer rows are live in L2 at once (kClu below).
//
// A CTA is warp-specialised. One producer warp streams the row in chunks
// (bulk async copies, non-multicast) into a ring of shared-memory slots,
// each slot with a "full" mbarrier (transaction bytes) and an "empty"
// mbarrier (one arrival per consumer warp). The producer walks the task list
// row by row: the chunks of the row for pass A, then, for pass B, the same
// chunks in reverse order except the last, which pass B takes from the slot
// pass A left it in (the consumers release that slot only after pass B has
// used it). Pass A's copies of chunks that are read again are marked
// evict-last in L2, every other copy evict-first: with one CTA per SM only
// ~one row per SM is live (~46 MB on the headline workload, against a
// 126 MB L2), so the second read of a row is served by L2 and HBM sees each
// logit about once (checked with the DRAM byte counters); the reverse order
// re-reads the most recently copied chunk first. The consumer warps:
//   pass A  per chunk, each thread sums its vectors into (S, U) in packed
//           f32x2 against a running reference that moves by whole powers of
//           two (no per-element maximum), then releases the slot;
//   merge   butterfly merges, largest reference first, in a fixed order;
//           with top-K OPD on, warp 0 also takes the row's top-K part from
//           the top-K warp (one more warp, which gathers the candidates from
//           the ring slots as pass A's chunks arrive);
//   epilogue one thread evaluates the per-token objective and the gradient
//           coefficients;
//   pass B  per chunk, last to first, dLogits from the chunk, 16-byte streaming
//           stores; the sampled token's entry is rewritten during the next
//           row's epilogue (after a barrier that orders every store before it).
// Definitions: Sec. 3.4 (ratio), Sec. 2 / 9.1 (advantage), Sec. 2.4 (mask).
#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "kernels.h"
#include "stream_plan.h"

namespace milesloss {

namespace {

constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr float kLn2f = 0.69314718055994531f;

// Named barrier 1 among the kCW consumer warps of the CTA.
template <int kCW>
__device__ __forceinline__ void cons_sync() {
  asm volatile("bar.sync 1, %0;" ::"r"(kCW * 32) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// A thread's (or a group's) partial sums over a row, against a reference r
// in log2 units (a multiple of k = log2(e) / T of a logit):
//   s = sum_j 2^(z_j k - r),  u = sum_j 2^(z_j k - r) (z_j k - r).
// Any finite r gives the same row statistics: lse = r ln 2 + ln s and
// H = ln s - u ln 2 / s.
struct Tri {
  float m, s, u;  // m = r
};

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

// Merges the kCW consumer warps' partial sums of a row: red[w] = (m, s, u)
// of warp w, redm[w] = its m again (contiguous, so that every lane takes the
// maximum with kCW / 4 broadcast reads instead of a shuffle tree). Lanes
// 0..kCW-1 rescale one warp's sums each and sum them in a fixed order (xor
// butterflies within each group of kCW lanes); lane 0 gets the row's sums.
template <int kCW>
__device__ __forceinline__ Tri block_merge(const float4* red, const float* redm, int lane) {
  static_assert(kCW % 4 == 0 && kCW <= 32, "whole float4 of references, one warp of lanes");
  float M = -INFINITY;
#pragma unroll
  for (int w = 0; w < kCW / 4; ++w) {
    const float4 m4 = reinterpret_cast<const float4*>(redm)[w];
    M = fmaxf(M, fmaxf(fmaxf(m4.x, m4.y), fmaxf(m4.z, m4.w)));
  }
  float s = 0.0f, u = 0.0f;
  if (lane < kCW) {
    const float4 v = red[lane];
    if (v.y > 0.0f) {
      const float d = v.x - M, f = ex2(d);
      s = f * v.y;
      u = f * fmaf(d, v.y, v.z);
    }
  }
#pragma unroll
  for (int o = kCW / 2; o > 0; o >>= 1) {
    s += __shfl_xor_sync(0xffffffffu, s, o);
    u += __shfl_xor_sync(0xffffffffu, u, o);
  }
  return Tri{M, s, u};
}

// Running sums of one thread over the chunks of a row. The reference starts
// at the maximum of the thread's first vector and is moved only by whole
// powers of two of the sums (rebase), so no per-element maximum is needed.
struct Run {
  float r = -INFINITY;
  float2 s0 = {0.0f, 0.0f}, s1 = {0.0f, 0.0f}, u0 = {0.0f, 0.0f}, u1 = {0.0f, 0.0f};

  // move the reference up to nr (sums rescaled by 2^(r - nr))
  __device__ __forceinline__ void raise(float nr) {
    if (!(nr > r)) return;
    if (r != -INFINITY) {
      const float d = r - nr, f = ex2(d);
      const float2 f2 = make_float2(f, f), d2 = make_float2(d, d);
      u0 = fmul2(f2, ffma2(d2, s0, u0));
      u1 = fmul2(f2, ffma2(d2, s1, u1));
      s0 = fmul2(f2, s0);
      s1 = fmul2(f2, s1);
    }
    r = nr;
  }
  // After a chunk whose sums are finite: when they exceed 2^16, move the
  // reference up by their binary exponent e (s scales by 2^-e exactly).
  __device__ __forceinline__ void rebase() {
    const float2 s = fadd2(s0, s1);
    const int e = ((__float_as_int(s.x + s.y) >> 23) & 0xff) - 127;
    if (e > 16) {
      const float f = __int_as_float((127 - e) << 23), d = -static_cast<float>(e);
      const float2 f2 = make_float2(f, f), d2 = make_float2(d, d);
      u0 = fmul2(f2, ffma2(d2, s0, u0));
      u1 = fmul2(f2, ffma2(d2, s1, u1));
      s0 = fmul2(f2, s0);
      s1 = fmul2(f2, s1);
      r -= d;
    }
  }
  template <bool kSafe>
  __device__ __forceinline__ void add_pair(float2 z, float2 k2, float2& s, float2& u) {
    float2 t = ffma2(z, k2, make_float2(-r, -r));
    if (kSafe) {
      if (z.x == -INFINITY) t.x = -127.0f;
      if (z.y == -INFINITY) t.y = -127.0f;
    }
    const float2 x = ex2x2(t);
    s = fadd2(s, x);
    u = ffma2(x, t, u);
  }
  __device__ __forceinline__ Tri tri() const {
    const float2 s = fadd2(s0, s1), u = fadd2(u0, u1);
    return Tri{r, s.x + s.y, u.x + u.y};
  }
};

// dLogits of one chunk with vector stores. kMode 0: p ca with |ca| folded
// into the exponent; 1: the same negated; 2: p (ca + cb z).
template <class In, class Out, int kMode, int kCons>
__device__ __forceinline__ void pass_b_chunk(const uint4* sv, int nv, char* dchunk, float2 k2,
                                             float2 off2, float2 ca2, float2 cb2) {
  constexpr int V8 = In::kVec;
  constexpr int P = V8 / 2;
#pragma unroll 2
  for (int v = threadIdx.x; v < nv; v += kCons) {
    float2 f[P];
    In::unpack2(sv[v], f);
#pragma unroll
    for (int e = 0; e < P; ++e) {
      if (kMode == 2) {
        f[e] = fmul2(ex2x2(ffma2(f[e], k2, off2)), ent_factor2(f[e], ca2, cb2));
      } else {
        f[e] = ex2x2(ffma2(f[e], k2, off2));
        if (kMode == 1) f[e] = make_float2(-f[e].x, -f[e].y);
      }
    }
    Out::template storev<V8>(dchunk + static_cast<size_t>(v) * V8 * Out::kSize,
                             reinterpret_cast<const float*>(f), 0u);
  }
}

// kCW consumer warps: 16 with one CTA per SM, 8 with two, 4 with four (each
// CTA then has a half or a quarter of the SM's shared memory for its ring,
// and one CTA's per-row merge and epilogue overlap the others' passes).
//
// kClu (fused calls, sixteen consumer warps, no top-K, no vocabulary-shard
// records): the kernel runs in clusters of C CTAs, one cluster per row, CTA
// crank streaming the vectors [crank slice_vec, (crank + 1) slice_vec) of the
// row (the last CTA also the elements past the last whole vector) through its
// own ring. After pass A each CTA's thread 0 pushes the CTA's (m, s, u, z_y)
// into every peer's shared memory (st.async, counted on the peer's mbarrier
// for that row parity) and merges the C entries in rank order, so every CTA
// of the cluster holds the same row statistics and gradient coefficients;
// then each CTA writes its part of the row's dLogits. With C CTAs per row,
// C times fewer rows are live at once, so a long row's second read still
// comes from L2 (one CTA per SM keeps 152 rows live: 78 MB of 512 KB rows,
// 304 MB of 2 MB rows, against a 126 MB L2).
template <class In, class Out, bool kGrad, bool kTopK, int kCW, bool kClu>
__global__ void __launch_bounds__(kCW * 32 + (kTopK ? 64 : 32), 16 / kCW) k_stream(const StreamArgs a) {
  static_assert(!kClu || (kGrad && !kTopK && kCW == 16), "clusters: fused calls without top-K");
  constexpr int kCons = kCW * 32;  // consumer threads
  constexpr int kConsWarps = kCW;
  using St = typename In::storage;
  constexpr int V8 = In::kVec;
  constexpr int P = V8 / 2;
  extern __shared__ __align__(128) unsigned char smem[];
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int NS = a.n_slots;
  const int CB = a.chunk_bytes;
  const int CV = CB / 16;                        // vectors per full chunk
  // rows are visited by one CTA each (cl_id = the CTA) or by one cluster each
  const int C = kClu ? static_cast<int>(cluster_nctarank()) : 1;
  const int crank = kClu ? static_cast<int>(cluster_ctarank()) : 0;
  const long long cl_id = kClu ? blockIdx.x / C : blockIdx.x;
  const long long n_cl = kClu ? gridDim.x / C : gridDim.x;
  const int all_vec = a.V / V8;                  // whole 16-byte vectors per row
  const int lo_v = kClu ? min(all_vec, crank * a.slice_vec) : 0;  // this CTA's first vector
  const int row_vec = kClu ? min(all_vec - lo_v, a.slice_vec) : all_vec;  // ... and count
  const int tail0 = all_vec * V8;                // first element not in a vector
  const int my_tail0 = (crank == C - 1) ? tail0 : a.V;  // this CTA's part of those
  const int n_chunks = (row_vec + CV - 1) / CV;
  // Chunk c starts at vector cs(c) and holds cn(c) vectors. With
  // split_first the first chunk takes the remainder, rounded up to a multiple
  // of 8 vectors (128 bytes) so that every later chunk starts 128-byte aligned
  // and the last chunks, which pass B takes from shared memory, are (nearly)
  // full; otherwise the last chunk is the ragged one.
  const int rem = row_vec - (n_chunks - 1) * CV;
  const int f0 = a.split_first ? min(CV, (rem + 7) & ~7) : CV;
  auto cs = [&](int c) { return c == 0 ? 0 : min(row_vec, f0 + (c - 1) * CV); };
  auto cn = [&](int c) { return cs(c + 1) - cs(c); };
  const float k = a.s.k;

  unsigned char* ring = smem;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(NS) * CB);
  uint64_t* empty = full + kMaxSlots;
  float4* red = reinterpret_cast<float4*>(empty + kMaxSlots);  // [kConsWarps]
  float* redm = reinterpret_cast<float*>(red + kConsWarps);     // [kConsWarps]
  float4* bc = reinterpret_cast<float4*>(redm + kConsWarps);    // [2]
  int4* bci = reinterpret_cast<int4*>(bc + 2);                  // [1]
  TopKPart* tkp = reinterpret_cast<TopKPart*>(bci + 1);         // [2] top-K parts by row parity
  uint64_t* tk_full = reinterpret_cast<uint64_t*>(tkp + 2);     // [2] part written
  uint64_t* tk_empty = tk_full + 2;                             // [2] part read
  uint64_t* never = tk_empty + 2;                               // [1] completed by nothing (test hook)
  volatile int* abort = reinterpret_cast<volatile int*>(never + 1);  // the CTA gave up
  uint64_t* xbar = never + 2;                                   // [2] exchange barriers (kClu)
  float4* xch = reinterpret_cast<float4*>(
      (reinterpret_cast<uintptr_t>(xbar + 2) + 15) & ~static_cast<uintptr_t>(15));  // [2][kMaxCluster]
  static_assert(2 * kMaxSlots * 8 + (kConsWarps + 3) * 16 + kConsWarps * 4 + 2 * sizeof(TopKPart) +
                        6 * 8 + 2 * 8 + 8 + 2 * kMaxCluster * 16 <=
                    kSweepSmemExtra,
                "k_stream scratch");
  // [2] top-K candidates of this row and the next (launched with kTopKSmem more)
  TopKBuf* tkb = reinterpret_cast<TopKBuf*>(smem + static_cast<size_t>(NS) * CB + kSweepSmemExtra);

  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), kConsWarps + (kTopK ? 1 : 0));
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&tk_full[b]), 1);
      mbar_init(smem_u32(&tk_empty[b]), 1);
    }
    mbar_init(smem_u32(never), 1);
    if (kClu) {
      mbar_init(smem_u32(&xbar[0]), 1);
      mbar_init(smem_u32(&xbar[1]), 1);
    }
    *abort = 0;
    fence_mbar_init();
  }
  // (peers push into this CTA's exchange slots: every barrier of the cluster
  // is initialised before any CTA goes on)
  if constexpr (kClu) cluster_sync_all();
  else __syncthreads();

  WsPtrs ws = a.ws;
  uint32_t* err = &ws.hdr->err_bits;
  const char* lg = static_cast<const char*>(a.logits);
  const long long rows_mine = (a.R > cl_id) ? (a.R - 1 - cl_id) / n_cl + 1 : 0;

  // Every wait below is bounded and, except the producer's waits for its own
  // copies, also ends as soon as another party of the CTA has given up
  // (mbar_wait_or_abort). After giving up, a party reads no ring slot it has
  // not waited for, keeps its arrivals (so no barrier is left short of
  // them), and the rows still to come are written as zeros.
  if (warp == kConsWarps) {
    // ------------------------------------------------------------ producer
    // A slot is re-armed only once every reader has released the task the
    // slot held. A reader that gave up on a wait releases its tasks without
    // reading them, but it raised the CTA's flag before its release (the
    // release orders that store before the arrival the producer's wait
    // observes), so after every completed wait the producer checks the flag
    // and, when it is up, issues nothing more: no copy is issued over one
    // still in flight or over data still being read. Before it returns, the
    // producer waits (bounded) for the last copy issued into each slot,
    // timeout or not, so no bulk copy lands in this CTA's shared memory after
    // the CTA exits.
    if (lane == 0) {
      const uint64_t pol_a = l2_policy_evict_last(), pol_b = l2_policy_evict_first();
      bool stop = false;
      long long q = 0;
      // each row's mask byte is loaded one row ahead, so that its latency
      // (often a DRAM access: a CTA's rows are n_cl bytes apart) never
      // delays the row it decides
      uint8_t mask_next = rows_mine > 0 ? a.mask[cl_id] : 0;
      for (long long i = 0; i < rows_mine && !stop; ++i) {
        const long long row = cl_id + i * n_cl;
        const char* src_row = lg + row * a.ld * static_cast<long long>(sizeof(St)) +
                              static_cast<long long>(lo_v) * 16;
        const uint8_t msk_row = mask_next;
        if (i + 1 < rows_mine) mask_next = a.mask[row + n_cl];
        // a row that does not train has an all-zero gradient: no second read
        const bool again = kGrad && msk_row && n_chunks > 0;
        const int h = again ? min(a.n_hold, n_chunks) : 0;
        const int tasks = again ? 2 * n_chunks - h : n_chunks;
        for (int t = 0; t < tasks; ++t, ++q) {
          // pass A: chunks 0 .. n-1; pass B: chunks n-h-1 .. 0 (the last h
          // stay in their slots)
          const int c = (t < n_chunks) ? t : 2 * n_chunks - h - 1 - t;
          const int s = static_cast<int>(q % NS);
          // every reader has released the task NS back (and none gave up)
          if (q >= NS && (!mbar_wait_or_abort(smem_u32(&empty[s]),
                                              static_cast<uint32_t>(((q / NS) - 1) & 1),
                                              kWaitLimitNs, abort, err) ||
                          *abort)) {
            stop = true;
            break;
          }
          const int v0 = cs(c);
          const uint32_t bytes = static_cast<uint32_t>(cn(c)) * 16u;
          const uint32_t bar = smem_u32(&full[s]);
          mbar_arrive_expect_tx(bar, bytes);
          bulk_g2s(smem_u32(ring + static_cast<size_t>(s) * CB), src_row + static_cast<size_t>(v0) * 16,
                   bytes, bar, (again && t < n_chunks - h) ? pol_a : pol_b);
          if (t == n_chunks - 1 && a.prefetch > 0 && i + 1 < rows_mine) {
            // the row's first pass is issued: ask L2 for the head of the next
            // row, so that HBM keeps reading while this row is merged
            const char* nxt = src_row + n_cl * a.ld * static_cast<long long>(sizeof(St));
            const uint32_t total = min(static_cast<uint32_t>(a.prefetch),
                                       static_cast<uint32_t>(row_vec) * 16u);
            for (uint32_t off = 0; off < total; off += 32768u)
              bulk_prefetch_l2(nxt + off, min(32768u, total - off));
          }
        }
      }
      // Wait (bounded) for the last copy issued into each slot before the
      // CTA can exit: returns at once when the readers already waited for it.
      for (int s = 0; s < NS; ++s) {
        if (q > s) {
          const long long last = q - 1 - ((q - 1 - s) % NS);
          if (!mbar_wait_bounded(smem_u32(&full[s]), static_cast<uint32_t>((last / NS) & 1),
                                 kWaitLimitNs))
            atomicOr(err, kErrTimeout);
        }
      }
    }
    if constexpr (kClu) {  // the cluster's closing barrier (every thread of every CTA)
      __syncwarp();
      cluster_sync_all();
    }
    return;
  }

  if (kTopK && warp == kConsWarps + 1) {
    // ------------------------------------------------------------- top-K OPD
    // One more warp takes each row's top-K candidate logits from the ring
    // slots as pass A's chunks arrive (it waits on every task's "full"
    // barrier and is one more arrival on its "empty" barrier) and computes the
    // candidates' part of the signal, which needs no row statistics, while the
    // consumers finish pass A; warp 0 takes the part after the merge. The
    // parts are double-buffered by row parity, each buffer with a "written"
    // and a "read" mbarrier (one arrival each), so this warp may run up to a
    // row ahead. (A named barrier synced by both warps once per row cost
    // ~1 us per row on GB300: 6.72 against 6.26 ms on 65,536 x 154,880.) The
    // row's ids and teacher values were copied during the previous row.
    auto twait = [&](long long q) {
      const int s = static_cast<int>(q % NS);
      const bool ok = mbar_wait_or_abort(smem_u32(&full[s]), static_cast<uint32_t>((q / NS) & 1),
                                         kWaitLimitNs, abort, err);
      return ok ? reinterpret_cast<const uint4*>(ring + static_cast<size_t>(s) * CB) : nullptr;
    };
    auto tarrive = [&](long long q) {
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&empty[q % NS]));
    };
    const int K = a.s.topk;
    if (rows_mine > 0)
      topk_prefetch(&tkb[0], a.s.topk_ids + cl_id * K, a.s.topk_teacher + cl_id * K, K, lane);
    long long q0 = 0;
    uint8_t mask_next = rows_mine > 0 ? a.mask[cl_id] : 0;  // one row ahead
    for (long long i = 0; i < rows_mine; ++i) {
      const long long row = cl_id + i * n_cl;
      const bool trains = mask_next != 0;
      if (i + 1 < rows_mine) mask_next = a.mask[row + n_cl];
      const int h = (kGrad && trains && n_chunks > 0) ? min(a.n_hold, n_chunks) : 0;
      const TopKBuf* tk_row = &tkb[i & 1];
      cp_async_wait_all();
      TopKLane tk = topk_ids(tk_row, static_cast<int>(a.col0), a.V, a.vocab_total, K, lane);
      if (i + 1 < rows_mine) {
        const long long o = (row + n_cl) * K;
        topk_prefetch(&tkb[(i + 1) & 1], a.s.topk_ids + o, a.s.topk_teacher + o, K, lane);
      }
      for (int c = 0; c < n_chunks; ++c) {
        const uint4* sv = twait(q0 + c);
        const int v0 = cs(c);
        if (sv) topk_gather<In>(tk, sv, v0 * V8, (v0 + cn(c)) * V8);
        tarrive(q0 + c);
      }
      if (tail0 < a.V)  // candidates past the last whole vector
        topk_gather<In>(tk, reinterpret_cast<const St*>(lg + row * a.ld * static_cast<long long>(sizeof(St))) + tail0,
                        tail0, a.V);
      const TopKPart p = topk_part(tk, tk_row, lane, a.s.invT, k, [](int) { return true; });
      // the part of row i - 2 (same buffer) has been read
      if (i >= 2)
        mbar_wait_or_abort(smem_u32(&tk_empty[i & 1]), static_cast<uint32_t>(((i >> 1) - 1) & 1),
                           kWaitLimitNs, abort, err);
      if (lane == 0) {
        tkp[i & 1] = p;
        mbar_arrive(smem_u32(&tk_full[i & 1]));
      }
      // pass B's copies: this warp's arrivals keep the slots' counts
      if (kGrad && trains) {
        for (int j = h; j < n_chunks; ++j) {
          const long long qq = q0 + n_chunks + (j - h);
          twait(qq);
          tarrive(qq);
        }
      }
      q0 += (kGrad && trains) ? 2 * n_chunks - h : n_chunks;
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  const long long N = ws.hdr->n_tokens;
  float g = a.grad_loss;
  if (a.grad_loss_dev) g *= *a.grad_loss_dev;
  const float cscale = (N > 0) ? g / static_cast<float>(N) * a.s.invT : 0.0f;
  const float2 k2 = make_float2(k, k);
  // the sampled token's dLogit of the previous row, written after the next
  // barrier (so after every store of that row)
  char* fix_ptr = nullptr;
  float fix_val = 0.0f;

  // Waits for task q's copy; false: this thread gave up (the CTA's flag is
  // up). Pass A reads the slot either way (reading shared memory that a copy
  // may still be writing is harmless, and the epilogue then writes the row
  // as zeros); pass B writes zeros instead.
  auto wait_slot = [&](long long q) {
    return mbar_wait_or_abort(smem_u32(&full[q % NS]), static_cast<uint32_t>((q / NS) & 1),
                              kWaitLimitNs, abort, err);
  };
  auto slot = [&](long long q) {
    return reinterpret_cast<const uint4*>(ring + static_cast<size_t>(q % NS) * CB);
  };
  auto release_slot = [&](long long q) {
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&empty[q % NS]));
  };

  if (a.stall_ns) {
    // test hook: a wait on a barrier that nothing completes, before the
    // first row; it runs out and raises the flag, so every wait after it
    // gives up at once
    mbar_wait_or_abort(smem_u32(never), 0u, a.stall_ns, abort, err);
  }

  long long q0 = 0;  // task number of the row's first chunk (same count as the producer's)
  bool xdead = false;  // (kClu, thread 0) an exchange wait of this CTA ran out
  uint8_t mask_next = rows_mine > 0 ? a.mask[cl_id] : 0;  // one row ahead
  for (long long i = 0; i < rows_mine; ++i) {
    const long long row = cl_id + i * n_cl;
    const char* grow = lg + row * a.ld * static_cast<long long>(sizeof(St));
    const bool trains = mask_next != 0;
    if (i + 1 < rows_mine) mask_next = a.mask[row + n_cl];
    // pass B takes the last h chunks from the slots pass A left them in
    const int h = (kGrad && trains && n_chunks > 0) ? min(a.n_hold, n_chunks) : 0;

    int y = 0;
    float rho = 0.0f, q = 0.0f, old = 0.0f, A = 0.0f, zy = 0.0f;
    uint8_t msk = 0;
    bool yok = false;
    if (tid == 0) {
      // the target's column in this call's logits (-1 outside them: a bad
      // target, or another shard's column in a vocabulary-sharded call)
      const long long yl = a.targets[row] - a.col0;
      y = (yl >= 0 && yl < a.V) ? static_cast<int>(yl) : -1;
      rho = a.rho[row];
      if (a.q) q = a.q[row];
      if (a.old) old = a.old[row];
      A = ws.a_row[row];
      msk = trains ? 1 : 0;
      yok = y >= 0;
      if (yok && y >= my_tail0) zy = In::load1(grow, y);
    }
    // the target's vector within this CTA's vectors, and (kClu) the CTA
    // whose part of the row holds the target (thread 0 only)
    const int yv = yok ? y / V8 - lo_v : -1;
    const int owner = (!kClu || !yok) ? 0 : (y >= tail0 ? C - 1 : min(C - 1, (y / V8) / a.slice_vec));

    // ---------------- pass A
    // One sweep of each chunk in shared memory against the thread's running
    // reference (for the first chunk, the maximum of the thread's first
    // vector): the sums are finite unless a logit lies more than 127 / k
    // above the reference, and that case (an overflow, seen as inf) or a
    // -inf logit (NaN) redoes the chunk against the chunk's own maximum,
    // skipping -inf logits exactly.
    Run run;
    for (int c = 0; c < n_chunks; ++c) {
      wait_slot(q0 + c);
      const uint4* sv = slot(q0 + c);
      const int v0 = cs(c), nv = cn(c);
      {
        if (tid == 0 && yv >= v0 && yv < v0 + nv) zy = In::load1(sv, y - (lo_v + v0) * V8);
        if (run.r == -INFINITY && tid < nv) run.raise(In::vmax(sv[tid]) * k);
        const Run keep = run;
        bool redo = run.r == -INFINITY;  // no finite reference yet
        if (!redo) {
#pragma unroll 4
          for (int v = tid; v < nv; v += kCons) {
            float2 f[P];
            In::unpack2(sv[v], f);
#pragma unroll
            for (int e = 0; e < P; ++e) run.add_pair<false>(f[e], k2, (e & 1) ? run.s1 : run.s0,
                                                            (e & 1) ? run.u1 : run.u0);
          }
          const Tri cur = run.tri();
          redo = !(fabsf(cur.s) < INFINITY) || !(fabsf(cur.u) < INFINITY);  // inf or NaN
          if (!redo) run.rebase();
        }
        if (redo) {
          typename In::MaxAcc macc = In::kMaxInit;
          for (int v = tid; v < nv; v += kCons) macc = In::max_acc(macc, sv[v]);
          run = keep;
          run.raise(In::max_val(macc) * k);
          if (run.r != -INFINITY) {
            for (int v = tid; v < nv; v += kCons) {
              float2 f[P];
              In::unpack2(sv[v], f);
#pragma unroll
              for (int e = 0; e < P; ++e) run.add_pair<true>(f[e], k2, run.s0, run.u0);
            }
          }
        }
      }
      if (c < n_chunks - h) release_slot(q0 + c);
    }
    Tri t = run.tri();
    for (int j = my_tail0 + tid; j < a.V; j += kCons) {
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

    // ---------------- merge
    t = warp_merge(t);
    if (lane == 0) {
      red[warp] = make_float4(t.m, t.s, t.u, 0.0f);
      redm[warp] = t.m;
    }
    cons_sync<kCW>();
    if (tid == 0 && fix_ptr) Out::store1(fix_ptr, 0, fix_val);  // previous row's y entry
    fix_ptr = nullptr;
    if (warp == 0) t = block_merge<kCW>(red, redm, lane);
    bool cl_bad = false;  // (kClu, thread 0) a CTA of the cluster gave up before this row
    if constexpr (kClu) {
      if (tid == 0) {
        // the cluster's row statistics: this CTA's (m, s, u, z_y) into every
        // peer's slot for this row parity, then the C entries merged in rank
        // order (the same bits in every CTA). A CTA whose wait ran out keeps
        // pushing but waits no more (its rows are written as zeros).
        const int slot = static_cast<int>(i & 1);
        float4* xs = xch + slot * kMaxCluster;
        // (s = -1, which no row's sums take, marks a CTA that gave up)
        const float4 mine = make_float4(t.m, *abort ? -1.0f : t.s, t.u, zy);
        xs[crank] = mine;
        const uint32_t xaddr = smem_u32(&xs[crank]), xb = smem_u32(&xbar[slot]);
        for (int r = 0; r < C; ++r)
          if (r != crank) st_async_f4(mapa_shared(xaddr, r), mine, mapa_shared(xb, r));
        if (!xdead) {
          mbar_arrive_expect_tx(xb, static_cast<uint32_t>(C - 1) * 16u);
          if (!mbar_wait_bounded(xb, static_cast<uint32_t>((i >> 1) & 1), kWaitLimitNs)) {
            xdead = true;
            *abort = 1;
            atomicOr(err, kErrTimeout);
          }
        }
        float M = -INFINITY;
        for (int r = 0; r < C; ++r) {
          M = fmaxf(M, xs[r].x);
          cl_bad |= xs[r].y < 0.0f;
        }
        Tri tot{M, 0.0f, 0.0f};
        for (int r = 0; r < C; ++r) {
          const float4 e = xs[r];
          if (e.y > 0.0f) {
            const float d = e.x - M, f = ex2(d);
            tot.s += f * e.y;
            tot.u += f * fmaf(d, e.y, e.z);
          }
        }
        zy = xs[owner].w;
        t = tot;
      }
    }
    // top-K OPD signal (Sec. 5.2), a fixed per-token reward: the top-K warp's
    // part of this row and the row's lse (warp 0)
    float opd = 0.0f;
    int tk_bad = 0;
    TopKPart part{-INFINITY, 0.0f, 0.0f, 0};  // (kept for a vocabulary shard's record)
    if (kTopK && warp == 0) {
      if (mbar_wait_or_abort(smem_u32(&tk_full[i & 1]), static_cast<uint32_t>((i >> 1) & 1),
                             kWaitLimitNs, abort, err)) {
        part = tkp[i & 1];
        opd = topk_value(part, fmaf(t.m, kLn2f, logf(t.s)));
        tk_bad = part.bad;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&tk_empty[i & 1]));
    }

    // ---------------- epilogue (thread 0)
    // Only what pass B needs comes before the barrier (the row's statistics,
    // the per-token objective and the gradient coefficients); the stores of
    // the row's outputs and the sampled token's entry come after it, while
    // the other warps start pass B.
    char* drow = kGrad ? static_cast<char*>(a.dlogits) +
                             row * a.ld_out * static_cast<long long>(Out::kSize)
                       : nullptr;
    bool bad = false;
    float logp = 0.0f, H = 0.0f, lse = 0.0f, cc = 0.0f;
    TokenTerms tt{};
    if (tid == 0 && a.part_rows) {
      // vocabulary-sharded forward: the row's partial sums over this
      // shard's columns and its top-K candidates' part (a row read after
      // the CTA gave up is marked NaN)
      a.part_rows[2 * row] = *abort ? make_float4(NAN, 0.0f, 0.0f, 0.0f)
                                    : make_float4(t.m, t.s, t.u, yok ? zy : 0.0f);
      a.part_rows[2 * row + 1] = make_float4(part.m, part.sw, part.acc, part.bad ? 1.0f : 0.0f);
    } else if (tid == 0) {
      // a row read after the CTA gave up, a bad target or a bad top-K
      // candidate: zeros
      bad = !yok || tk_bad || *abort || cl_bad;
      const float lnS = logf(t.s);
      lse = fmaf(t.m, kLn2f, lnS);  // the reference is in log2 units
      H = lnS - t.u * kLn2f / t.s;
      logp = zy * a.s.invT - lse;
      if (bad) { logp = 0.0f; H = 0.0f; }
      if (a.s.topk > 0 && !bad) A -= a.s.opd_coef * opd;
      tt = token_terms(logp, H, rho, q, a.q != nullptr, old, a.old != nullptr, A, a.s);
      if (bad) tt = TokenTerms{0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, kFlagBad};
      if (kGrad) {
        cc = (msk && !bad) ? cscale : 0.0f;
        const float ca = cc * (-tt.G + a.s.gamma * (H - lse));
        const float cb = cc * a.s.gamma * a.s.invT;
        const float L2 = t.m + __log2f(t.s);
        const bool zero = (cc == 0.0f) || (ca == 0.0f && cb == 0.0f);
        const bool fold = !zero && (cb == 0.0f);
        const float off = fold ? (__log2f(fabsf(ca)) - L2) : -L2;
        bc[0] = make_float4(off, ca, cb, 0.0f);
        bci[0] = make_int4(zero, fold, (fold && ca < 0.0f) ? 1 : 0, 0);
      }
    }
    cons_sync<kCW>();
    if (tid == 0 && !a.part_rows) {
      if (crank == 0) {  // (one CTA of a cluster writes the row's results)
        if (!yok) atomicOr(err, kErrTarget);
        if (tk_bad) atomicOr(err, kErrTopK);
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
      // (the CTA whose part of the row holds the target)
      if (kGrad && owner == crank && cc != 0.0f && !bci[0].x) {
        // cc [G (1 - p_y) + gamma p_y (log p_y + H)], 1 - p_y = -expm1(logp);
        // written after the next row's merge barrier, which orders it after
        // every store of this row
        fix_ptr = drow + static_cast<long long>(y) * Out::kSize;
        fix_val = cc * (tt.G * -expm1f(logp) + a.s.gamma * expf(logp) * (logp + H));
      }
    }

    // ---------------- pass B
    if (kGrad) {
      const float4 cf = bc[0];
      const int4 ci = bci[0];
      const float2 off2 = make_float2(cf.x, cf.x);
      const float2 ca2 = make_float2(cf.y, cf.y), cb2 = make_float2(cf.z, cf.z);
      const bool vec_out = a.out_vec != 0;
      for (int j = 0; j < n_chunks; ++j) {
        // chunks n-h .. n-1 are still in the slots of tasks q0 + n - h ..
        // q0 + n - 1 (a wait on a completed phase returns at once); then
        // tasks q0 + n .. q0 + 2n - h - 1 bring chunks n-h-1 .. 0
        const int c = (j < h) ? n_chunks - h + j : n_chunks - 1 - j;
        const long long qq = (j < h) ? q0 + n_chunks - h + j : q0 + n_chunks + (j - h);
        const int nv = cn(c);
        char* dchunk = drow + static_cast<long long>(lo_v + cs(c)) * V8 * Out::kSize;
        auto zero_chunk = [&]() {
          float zf[V8];
#pragma unroll
          for (int e = 0; e < V8; ++e) zf[e] = 0.0f;
          for (int v = tid; v < nv; v += kCons) {
            if (vec_out) Out::template storev<V8>(dchunk + static_cast<size_t>(v) * V8 * Out::kSize, zf, 0u);
            else for (int e = 0; e < V8; ++e) Out::store1(dchunk, v * V8 + e, 0.0f);
          }
        };
        if (ci.x) {
          // zero gradient: the chunk's data is not needed; a training row's
          // chunk was still copied, so its slot is waited on and released to
          // keep the ring in step with the producer
          if (trains) wait_slot(qq);
          zero_chunk();
          if (trains) release_slot(qq);
          continue;
        }
        if (!wait_slot(qq)) {  // this thread gave up: zeros, not the slot's data
          zero_chunk();
          release_slot(qq);
          continue;
        }
        const uint4* sv = slot(qq);
        if (vec_out) {
          if (!ci.y) pass_b_chunk<In, Out, 2, kCons>(sv, nv, dchunk, k2, off2, ca2, cb2);
          else if (ci.z) pass_b_chunk<In, Out, 1, kCons>(sv, nv, dchunk, k2, off2, ca2, cb2);
          else pass_b_chunk<In, Out, 0, kCons>(sv, nv, dchunk, k2, off2, ca2, cb2);
        } else {
          for (int v = tid; v < nv; v += kCons) {
            float2 f[P];
            In::unpack2(sv[v], f);
#pragma unroll
            for (int e = 0; e < P; ++e) {
              f[e] = ci.y ? ex2x2(ffma2(f[e], k2, off2))
                          : fmul2(ex2x2(ffma2(f[e], k2, off2)), ent_factor2(f[e], ca2, cb2));
              if (ci.y && ci.z) f[e] = make_float2(-f[e].x, -f[e].y);
            }
            const float* fv = reinterpret_cast<const float*>(f);
            for (int e = 0; e < V8; ++e) Out::store1(dchunk, v * V8 + e, fv[e]);
          }
        }
        release_slot(qq);
      }
      for (int j = my_tail0 + tid; j < a.V; j += kCons) {
        const float z = In::load1(grow, j);
        float x = 0.0f;
        if (!ci.x) {
          x = ci.y ? ex2(fmaf(z, k, cf.x)) : ex2(fmaf(z, k, cf.x)) * ent_factor(z, cf.y, cf.z);
          if (ci.y && ci.z) x = -x;
        }
        Out::store1(drow, j, x);
      }
    }
    q0 += (kGrad && trains) ? 2 * n_chunks - h : n_chunks;
  }
  cons_sync<kCW>();
  if (tid == 0 && fix_ptr) Out::store1(fix_ptr, 0, fix_val);
  if constexpr (kClu) {  // no CTA leaves while a peer's last exchange store into it may be in flight
    __syncwarp();
    cluster_sync_all();
  }
}

template <class In, class Out, bool kGrad>
const void* fn(bool topk, int cw, bool clu) {
  if constexpr (kGrad) {
    if (clu) return topk ? nullptr : reinterpret_cast<const void*>(&k_stream<In, Out, true, false, 16, true>);
  } else {
    if (clu) return nullptr;
  }
  if (cw == 4)
    return topk ? reinterpret_cast<const void*>(&k_stream<In, Out, kGrad, true, 4, false>)
                : reinterpret_cast<const void*>(&k_stream<In, Out, kGrad, false, 4, false>);
  if (cw == 8)
    return topk ? reinterpret_cast<const void*>(&k_stream<In, Out, kGrad, true, 8, false>)
                : reinterpret_cast<const void*>(&k_stream<In, Out, kGrad, false, 8, false>);
  return topk ? reinterpret_cast<const void*>(&k_stream<In, Out, kGrad, true, 16, false>)
              : reinterpret_cast<const void*>(&k_stream<In, Out, kGrad, false, 16, false>);
}

}  // namespace

bool use_stream(long long row_bytes, int es, bool in_bulk, bool grad, bool topk,
                const rl_launch_overrides& ov) {
  if (ov.sweep_kernel == 0) return false;
  if (ov.sweep_kernel == 1) return in_bulk;
  return in_bulk && stream_ctas(row_bytes, es, grad, topk) > 0;
}

rl_status plan_stream(int dev, int extra, long long row_bytes, int es, bool grad, bool topk,
                      bool can_cluster, const rl_launch_overrides& ov, StreamPlan* out) {
  int optin = 0, per_sm = 0, reserved = 0;
  if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev) !=
          cudaSuccess)
    return RL_ERR_CUDA;
  return plan_stream_rows(row_bytes, es, grad, topk, can_cluster,
                          SmemLimits{optin, per_sm, reserved}, extra, ov, out)
             ? RL_OK
             : RL_ERR_UNSUPPORTED;
}

const void* stream_kernel(rl_dtype in, rl_dtype out, bool grad, bool topk, int cw, bool clu) {
  if (!grad)
    return in == RL_BF16 ? fn<InBf16, OutBf16, false>(topk, cw, clu)
                         : fn<InF32, OutF32, false>(topk, cw, clu);
  if (in == RL_BF16)
    return out == RL_BF16 ? fn<InBf16, OutBf16, true>(topk, cw, clu)
                          : fn<InBf16, OutF32, true>(topk, cw, clu);
  return out == RL_BF16 ? fn<InF32, OutBf16, true>(topk, cw, clu)
                        : fn<InF32, OutF32, true>(topk, cw, clu);
}

}  // namespace milesloss

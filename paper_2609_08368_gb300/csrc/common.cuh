// Device helpers and the workspace layout shared by the kernels of
// libmilesloss. sm_103a only: inline PTX for mbarrier, bulk async copies
// (cp.async.bulk, non-multicast), thread-block-cluster barriers and
// distributed shared memory.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "milesloss.h"

namespace milesloss {

// ------------------------------------------------------------------ errors
// Data-dependent errors are recorded as bits (1 << status code) in the
// workspace header; the host reports the lowest set code.
enum : uint32_t {
  kErrTarget = 1u << RL_ERR_TARGET_OUT_OF_RANGE,
  kErrGroup = 1u << RL_ERR_GROUP_OUT_OF_RANGE,
  kErrSeqlens = 1u << RL_ERR_BAD_SEQLENS,
  kErrTimeout = 1u << RL_ERR_DEVICE_TIMEOUT,
  kErrTopK = 1u << RL_ERR_TOPK_ID_OUT_OF_RANGE,
};

// Per-row flag bits kept in the workspace.
enum : uint8_t {
  kFlagClipHi = 1, kFlagClipLo = 2, kFlagDual = 4, kFlagCorrClip = 8, kFlagBad = 16,
};

// --------------------------------------------------------------- workspace
struct WsHeader {
  uint32_t err_bits;   // OR of kErr* bits
  uint32_t ticket;     // last-block counter of the statistics reduction
  long long n_tokens;  // N = sum of the loss mask, written by the advantage kernel
  long long n_seq;     // trajectories with at least one training token
  uint32_t pad[58];
};
static_assert(sizeof(WsHeader) == 256, "header is one 256-byte segment");

// Partial sums of one block of the statistics reduction.
struct StatPart {
  double s_ell, s_pg, s_k3, s_H, s_r, s_rabs, s_lpabs, s_rc, s_rcabs;
  float rmin, rmax;
  unsigned long long n, n_hi, n_lo, n_dual, n_corr;
};

constexpr int kMaxTopK = 64;
constexpr int kStatThreads = 256;
constexpr int kMaxStatBlocks = 256;  // one partial per thread of the final block

struct WsLayout {
  size_t hdr, g_mu, g_den, g_flag, a_traj, traj_n, a_row;
  size_t r_logp, r_H, r_lse, r_G, r_ell, r_pg, r_k3, r_r, r_rc, r_flags;
  size_t parts, total;

  __host__ __device__ static size_t up(size_t x) { return (x + 255) & ~size_t(255); }

  // Per-row state first: its offsets depend on the row count only, so the
  // backward call (which does not know the trajectory and group counts)
  // finds it.
  __host__ __device__ static WsLayout make(long long R, int n_traj, int n_groups) {
    WsLayout L;
    size_t o = 0;
    L.hdr = o; o += up(sizeof(WsHeader));
    L.a_row = o; o += up(sizeof(float) * (size_t)R);
    size_t* rows[] = {&L.r_logp, &L.r_H, &L.r_lse, &L.r_G, &L.r_ell,
                      &L.r_pg, &L.r_k3, &L.r_r, &L.r_rc};
    for (size_t* p : rows) { *p = o; o += up(sizeof(float) * (size_t)R); }
    L.r_flags = o; o += up((size_t)R);
    L.parts = o; o += up(sizeof(StatPart) * kMaxStatBlocks);
    L.g_mu = o; o += up(sizeof(double) * (size_t)n_groups);
    L.g_den = o; o += up(sizeof(double) * (size_t)n_groups);
    L.g_flag = o; o += up(sizeof(int) * (size_t)n_groups);
    L.a_traj = o; o += up(sizeof(float) * (size_t)n_traj);
    L.traj_n = o; o += up(sizeof(int) * (size_t)n_traj);
    L.total = o;
    return L;
  }
};

// Pointers into one workspace.
struct WsPtrs {
  WsHeader* hdr;
  double* g_mu;
  double* g_den;
  int* g_flag;
  float* a_traj;
  int* traj_n;  // training tokens per trajectory
  float* a_row;
  float *logp, *H, *lse, *G, *ell, *pg, *k3, *r, *rc;
  uint8_t* flags;
  StatPart* parts;

  static WsPtrs at(void* base, const WsLayout& L) {
    char* b = static_cast<char*>(base);
    WsPtrs p;
    p.hdr = reinterpret_cast<WsHeader*>(b + L.hdr);
    p.g_mu = reinterpret_cast<double*>(b + L.g_mu);
    p.g_den = reinterpret_cast<double*>(b + L.g_den);
    p.g_flag = reinterpret_cast<int*>(b + L.g_flag);
    p.a_traj = reinterpret_cast<float*>(b + L.a_traj);
    p.traj_n = reinterpret_cast<int*>(b + L.traj_n);
    p.a_row = reinterpret_cast<float*>(b + L.a_row);
    p.logp = reinterpret_cast<float*>(b + L.r_logp);
    p.H = reinterpret_cast<float*>(b + L.r_H);
    p.lse = reinterpret_cast<float*>(b + L.r_lse);
    p.G = reinterpret_cast<float*>(b + L.r_G);
    p.ell = reinterpret_cast<float*>(b + L.r_ell);
    p.pg = reinterpret_cast<float*>(b + L.r_pg);
    p.k3 = reinterpret_cast<float*>(b + L.r_k3);
    p.r = reinterpret_cast<float*>(b + L.r_r);
    p.rc = reinterpret_cast<float*>(b + L.r_rc);
    p.flags = reinterpret_cast<uint8_t*>(b + L.r_flags);
    p.parts = reinterpret_cast<StatPart*>(b + L.parts);
    return p;
  }
};

// Scalar parameters as the kernels use them.
struct LossScalars {
  float invT;      // 1 / T
  float k;         // log2(e) / T: logits -> base-2 exponent units
  float eps_lo, eps_hi, dual_c, beta, gamma, corr_lo, corr_hi;
  int corr;        // rl_correction
  int topk;        // K of the top-K OPD signal applied in the sweep epilogue (0 = none)
  float opd_coef;
  const int* topk_ids;       // [R, K]
  const float* topk_teacher; // [R, K]
};

// Correction weight of a token (Sec. 3.4) from its train/rollout ratio rc.
__host__ __device__ __forceinline__ float correction_weight(float rc, const LossScalars& s) {
  if (s.corr == RL_CORR_NONE) return 1.0f;
  if (s.corr == RL_CORR_TIS) return fminf(fmaxf(rc, s.corr_lo), s.corr_hi);
  return (rc < s.corr_lo || rc > s.corr_hi) ? 0.0f : rc;
}

// ------------------------------------------------------------------ PTX
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ float ex2(float x) {  // 2^x, flush-to-zero
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Waits for the phase with the given parity; gives up after ~limit_ns.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity,
                                                  uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t n = 1;; ++n) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((n & 63u) == 0 && globaltimer_ns() - t0 > limit_ns) return false;
  }
}

// A CTA's shared "give up" flag: once one party of the CTA has given up on a
// wait, the others stop waiting too (their next wait returns at once), so a
// CTA that meets one timeout finishes in about one wait limit instead of one
// limit per remaining wait.
//
// Waits for the phase with the given parity. Returns false without waiting
// when *abort is already set, and gives up when *abort becomes set or after
// ~limit_ns; a party that gives up on its own time limit records the timeout
// in *err. On false the caller must not read what the phase guards. Every
// party that returns false (re)sets *abort itself, so that whoever it later
// synchronises with (a barrier, an mbarrier arrival) sees the flag.
__device__ __forceinline__ bool mbar_wait_or_abort(uint32_t bar, uint32_t parity,
                                                   uint64_t limit_ns, volatile int* abort,
                                                   uint32_t* err) {
  // the flag is read first: a party that runs on after giving up must not
  // trust a parity test, which a barrier two phases behind would pass (the
  // flag load and the first test are independent, so their latencies overlap)
  const int gave_up = *abort;
  const bool done = mbar_try_wait(bar, parity);
  if (gave_up) {
    *abort = 1;
    return false;
  }
  if (done) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t n = 1;; ++n) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((n & 63u) == 0) {
      if (*abort) {
        *abort = 1;
        return false;
      }
      if (globaltimer_ns() - t0 > limit_ns) {
        *abort = 1;
        atomicOr(err, kErrTimeout);
        return false;
      }
    }
  }
}

__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// Global -> own shared memory bulk copy (no multicast); completion is
// signalled on the mbarrier as transaction bytes. dst, src 16-byte aligned;
// bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                         uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar), "l"(policy)
      : "memory");
}

// Asks L2 to fetch [src, src + bytes) from global memory (no destination, no
// completion to wait for). src 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint32_t cluster_nctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

__device__ __forceinline__ float4 ld_dsmem_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// Asynchronous 16-byte store into the shared memory of a CTA of the cluster
// (possibly another SM); the bytes are counted as transactions on the
// destination CTA's mbarrier. Both addresses come from mapa.
__device__ __forceinline__ void st_async_f4(uint32_t remote_addr, float4 v, uint32_t remote_bar) {
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];"
      ::"r"(remote_addr), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(remote_bar)
      : "memory");
}

// Packed pairs of fp32 (sm_100+ f32x2 instructions: two IEEE operations,
// each rounded to nearest, per instruction).
__device__ __forceinline__ unsigned long long f2_bits(float2 v) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(v.x), "f"(v.y));
  return r;
}
__device__ __forceinline__ float2 bits_f2(unsigned long long r) {
  float2 v;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(v.x), "=f"(v.y) : "l"(r));
  return v;
}
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  unsigned long long d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(f2_bits(a)), "l"(f2_bits(b)), "l"(f2_bits(c)));
  return bits_f2(d);
}
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
  unsigned long long d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(f2_bits(a)), "l"(f2_bits(b)));
  return bits_f2(d);
}
__device__ __forceinline__ float2 fmul2(float2 a, float2 b) {
  unsigned long long d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(f2_bits(a)), "l"(f2_bits(b)));
  return bits_f2(d);
}
__device__ __forceinline__ float2 ex2x2(float2 t) { return make_float2(ex2(t.x), ex2(t.y)); }

// The entropy term's factor (ca + cb z) of a logit z. A logit of -inf has
// probability zero and its p (ca + cb z) must be 0, not 0 * inf: the factor
// takes z no lower than kZFloor, far below any logit whose probability is
// not zero, where the vanishing p makes the product 0 whatever the floor.
constexpr float kZFloor = -1.0e20f;
__device__ __forceinline__ float ent_factor(float z, float ca, float cb) {
  return fmaf(cb, fmaxf(z, kZFloor), ca);
}
__device__ __forceinline__ float2 ent_factor2(float2 z, float2 ca2, float2 cb2) {
  return ffma2(cb2, make_float2(fmaxf(z.x, kZFloor), fmaxf(z.y, kZFloor)), ca2);
}

// Streaming 16-byte global load that does not allocate in L1.
__device__ __forceinline__ uint4 ld_stream_u4(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Streaming (evict-first) stores.
__device__ __forceinline__ void st_stream_u4(void* p, uint4 v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}
__device__ __forceinline__ void st_stream_u2(void* p, uint2 v) {
  asm volatile("st.global.cs.v2.u32 [%0], {%1, %2};" ::"l"(p), "r"(v.x), "r"(v.y) : "memory");
}

// ------------------------------------------------------------ dtype traits
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

struct InBf16 {
  using storage = uint16_t;
  static constexpr int kVec = 8;  // elements per 16 bytes
  __device__ static __forceinline__ void unpack(uint4 w, float* f) {
    f[0] = bf16_lo(w.x); f[1] = bf16_hi(w.x); f[2] = bf16_lo(w.y); f[3] = bf16_hi(w.y);
    f[4] = bf16_lo(w.z); f[5] = bf16_hi(w.z); f[6] = bf16_lo(w.w); f[7] = bf16_hi(w.w);
  }
  // the 16 bytes as kVec / 2 pairs
  __device__ static __forceinline__ void unpack2(uint4 w, float2* f) {
    f[0] = make_float2(bf16_lo(w.x), bf16_hi(w.x));
    f[1] = make_float2(bf16_lo(w.y), bf16_hi(w.y));
    f[2] = make_float2(bf16_lo(w.z), bf16_hi(w.z));
    f[3] = make_float2(bf16_lo(w.w), bf16_hi(w.w));
  }
  // running maximum kept as a packed pair (bf16x2 for bf16 input)
  using MaxAcc = uint32_t;
  static constexpr uint32_t kMaxInit = 0xff80ff80u;  // (-inf, -inf)
  __device__ static __forceinline__ uint32_t max_acc(uint32_t m, uint4 w) {
    __nv_bfloat162 a = __hmax2(*reinterpret_cast<__nv_bfloat162*>(&w.x),
                               *reinterpret_cast<__nv_bfloat162*>(&w.y));
    __nv_bfloat162 b = __hmax2(*reinterpret_cast<__nv_bfloat162*>(&w.z),
                               *reinterpret_cast<__nv_bfloat162*>(&w.w));
    __nv_bfloat162 c = __hmax2(__hmax2(a, b), *reinterpret_cast<__nv_bfloat162*>(&m));
    return *reinterpret_cast<uint32_t*>(&c);
  }
  __device__ static __forceinline__ float max_val(uint32_t m) {
    return fmaxf(bf16_lo(m), bf16_hi(m));
  }
  __device__ static __forceinline__ float vmax(uint4 w) {
    __nv_bfloat162 a = __hmax2(*reinterpret_cast<__nv_bfloat162*>(&w.x),
                               *reinterpret_cast<__nv_bfloat162*>(&w.y));
    __nv_bfloat162 b = __hmax2(*reinterpret_cast<__nv_bfloat162*>(&w.z),
                               *reinterpret_cast<__nv_bfloat162*>(&w.w));
    __nv_bfloat162 c = __hmax2(a, b);
    uint32_t u = *reinterpret_cast<uint32_t*>(&c);
    return fmaxf(bf16_lo(u), bf16_hi(u));
  }
  __device__ static __forceinline__ float load1(const void* base, long long i) {
    uint16_t h = static_cast<const uint16_t*>(base)[i];
    return __uint_as_float(static_cast<uint32_t>(h) << 16);
  }
};

struct InF32 {
  using storage = float;
  static constexpr int kVec = 4;
  __device__ static __forceinline__ void unpack(uint4 w, float* f) {
    f[0] = __uint_as_float(w.x); f[1] = __uint_as_float(w.y);
    f[2] = __uint_as_float(w.z); f[3] = __uint_as_float(w.w);
  }
  __device__ static __forceinline__ void unpack2(uint4 w, float2* f) {
    f[0] = make_float2(__uint_as_float(w.x), __uint_as_float(w.y));
    f[1] = make_float2(__uint_as_float(w.z), __uint_as_float(w.w));
  }
  using MaxAcc = float;
  static constexpr float kMaxInit = -INFINITY;
  __device__ static __forceinline__ float max_acc(float m, uint4 w) {
    return fmaxf(fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)),
                       fmaxf(__uint_as_float(w.z), __uint_as_float(w.w))), m);
  }
  __device__ static __forceinline__ float max_val(float m) { return m; }
  __device__ static __forceinline__ float vmax(uint4 w) {
    return fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)),
                 fmaxf(__uint_as_float(w.z), __uint_as_float(w.w)));
  }
  __device__ static __forceinline__ float load1(const void* base, long long i) {
    return static_cast<const float*>(base)[i];
  }
};

struct OutBf16 {
  static constexpr size_t kSize = 2;
  __device__ static __forceinline__ void store1(void* base, long long i, float v) {
    __nv_bfloat16 h = __float2bfloat16_rn(v);
    static_cast<__nv_bfloat16*>(base)[i] = h;
  }
  // n = 8 or 4 values starting at an element offset aligned to n * 2 bytes;
  // `sign` is XORed into every packed sign bit (0 or 0x80008000).
  template <int n>
  __device__ static __forceinline__ void storev(void* p, const float* f, uint32_t sign) {
    if constexpr (n == 8) {
      uint4 v = make_uint4(pack_bf16x2(f[0], f[1]) ^ sign, pack_bf16x2(f[2], f[3]) ^ sign,
                           pack_bf16x2(f[4], f[5]) ^ sign, pack_bf16x2(f[6], f[7]) ^ sign);
      st_stream_u4(p, v);
    } else {
      uint2 v = make_uint2(pack_bf16x2(f[0], f[1]) ^ sign, pack_bf16x2(f[2], f[3]) ^ sign);
      st_stream_u2(p, v);
    }
  }
  static constexpr uint32_t kSignMask = 0x80008000u;
};

struct OutF32 {
  static constexpr size_t kSize = 4;
  __device__ static __forceinline__ void store1(void* base, long long i, float v) {
    static_cast<float*>(base)[i] = v;
  }
  template <int n>
  __device__ static __forceinline__ void storev(void* p, const float* f, uint32_t sign) {
    uint4 a = make_uint4(__float_as_uint(f[0]) ^ sign, __float_as_uint(f[1]) ^ sign,
                         __float_as_uint(f[2]) ^ sign, __float_as_uint(f[3]) ^ sign);
    st_stream_u4(p, a);
    if constexpr (n == 8) {
      uint4 b = make_uint4(__float_as_uint(f[4]) ^ sign, __float_as_uint(f[5]) ^ sign,
                           __float_as_uint(f[6]) ^ sign, __float_as_uint(f[7]) ^ sign);
      st_stream_u4(static_cast<char*>(p) + 16, b);
    }
  }
  static constexpr uint32_t kSignMask = 0x80000000u;
};

// ------------------------------------------------- per-token objective
// The per-row epilogue shared by the fused and forward-only sweeps: from
// the row's log-prob and entropy, the token loss terms and G = dl/dlogp.
struct TokenTerms {
  float r, pg, k3, ell, G, rc;
  uint8_t flags;
};

// The policy-gradient part of a token's objective from its PPO ratio r and
// its correction ratio rc (Sec. 3.4; rc is ignored without a correction):
// pg (weighted by the correction), its derivative with respect to logp
// (weighted) and the clip flags.
struct PolicyTerms {
  float pg, gpg;
  uint8_t flags;
};

__device__ __forceinline__ PolicyTerms policy_terms(float r, float rc, float A,
                                                    const LossScalars& s) {
  const float u = -A * r;
  const float cl = fminf(fmaxf(r, 1.0f - s.eps_lo), 1.0f + s.eps_hi);
  const float c = -A * cl;
  const bool clipped = c > u;
  float pg = clipped ? c : u;
  uint8_t fl = 0;
  if (clipped && r > 1.0f + s.eps_hi) fl |= kFlagClipHi;
  if (clipped && r < 1.0f - s.eps_lo) fl |= kFlagClipLo;
  bool dual = false;
  if (s.dual_c > 0.0f && A < 0.0f) {
    const float d = -A * s.dual_c;
    if (d < pg) { pg = d; dual = true; fl |= kFlagDual; }
  }
  float gpg = (clipped || dual) ? 0.0f : -A * r;
  if (s.corr != RL_CORR_NONE) {
    if ((rc < s.corr_lo) || (rc > s.corr_hi)) fl |= kFlagCorrClip;
    const float wt = correction_weight(rc, s);
    pg *= wt;
    gpg *= wt;
  }
  return PolicyTerms{pg, gpg, fl};
}

__device__ __forceinline__ TokenTerms token_terms(float logp, float H, float rho, float q,
                                                  bool has_q, float old, bool has_old,
                                                  float A, const LossScalars& s) {
  TokenTerms t;
  const float base = has_old ? old : rho;
  const float r = expf(logp - base);
  // the train/rollout ratio of Sec. 3.4, log pi_train being the given old
  // log-prob or else this pass's own (then equal to r); a constant weight
  const float rc = s.corr == RL_CORR_NONE ? 1.0f : (has_old ? expf(old - rho) : r);
  const PolicyTerms pt = policy_terms(r, rc, A, s);
  float k3 = 0.0f, gkl = 0.0f;
  if (has_q) {
    // expm1 keeps both terms accurate when q is close to logp
    const float dlt = q - logp;
    const float em1 = expm1f(dlt);
    k3 = em1 - dlt;
    gkl = -em1;
  }
  t.r = r;
  t.pg = pt.pg;
  t.k3 = k3;
  t.ell = pt.pg + s.beta * k3 - s.gamma * H;
  t.G = pt.gpg + s.beta * gkl;
  t.rc = rc;
  t.flags = pt.flags;
  return t;
}

// Top-K on-policy distillation signal of one row (Sec. 5.2): the sum over
// the candidate set of w_k (log p_k - teacher_k), with p_k the trainer's
// probabilities of the candidates (from the row's logits and its lse) and
// w_k = p_k / sum_j p_j. A candidate outside [0, V) marks the row bad (it
// gets zeros and the call records RL_ERR_TOPK_ID_OUT_OF_RANGE).
//
// Since w_k is proportional to exp(z_k / T), the signal is
//   sum_k w_k (z_k / T - teacher_k) / sum_k w_k  -  lse,
// so partial sums over any subset of the candidates can be formed before lse
// is known and merged like the row statistics (a largest term, then sums
// rescaled to it): TopKPart below, with m the largest z_k k of the part (log2
// units, k = log2(e) / T, as the row statistics), sw = sum 2^(z_k k - m) and
// acc = sum 2^(z_k k - m)(z_k / T - teacher_k).
//
// One warp holds a row's candidates (K <= 64: lane l has candidates l and
// l + 32). Their ids and teacher log-probs are copied into shared memory one
// row ahead (cp.async: no registers held; each lane copies, and later reads,
// only its own entries). The candidates' logits are then taken from the copy
// of the row already in shared memory, which costs no DRAM access.
struct TopKBuf {
  int ids[kMaxTopK];
  float teacher[kMaxTopK];
};

struct TopKLane {
  int id0, id1;  // -1: no candidate (past K or outside [0, V))
  float z0, z1;
  bool bad;      // one of the lane's ids lies outside [0, V)
};

struct TopKPart {
  float m, sw, acc;
  int bad;  // some candidate id of the row lies outside [0, V)
};

__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_all;" ::: "memory");
}

__device__ __forceinline__ void topk_prefetch(TopKBuf* buf, const int* ids, const float* teacher,
                                              int K, int lane) {
  if (lane < K) {
    cp_async4(&buf->ids[lane], ids + lane);
    cp_async4(&buf->teacher[lane], teacher + lane);
  }
  if (lane + 32 < K) {
    cp_async4(&buf->ids[lane + 32], ids + lane + 32);
    cp_async4(&buf->teacher[lane + 32], teacher + lane + 32);
  }
  cp_async_commit();
}

// The lane's candidate ids of the row (after cp_async_wait_all for its
// buffer), as columns of this call's logits, which are the vocabulary's
// columns [col0, col0 + V) of a vocabulary of V_total (col0 = 0, V_total = V
// unless the call is a vocabulary shard): -1 for a candidate in another
// shard's columns; an id outside [0, V_total) marks the row bad.
__device__ __forceinline__ TopKLane topk_ids(const TopKBuf* buf, int col0, int V, int V_total,
                                             int K, int lane) {
  TopKLane c{-1, -1, 0.0f, 0.0f, false};
  if (lane < K) {
    const int id = buf->ids[lane];
    if (id < 0 || id >= V_total) c.bad = true;
    else if (id - col0 >= 0 && id - col0 < V) c.id0 = id - col0;
  }
  if (lane + 32 < K) {
    const int id = buf->ids[lane + 32];
    if (id < 0 || id >= V_total) c.bad = true;
    else if (id - col0 >= 0 && id - col0 < V) c.id1 = id - col0;
  }
  return c;
}

// Take the lane's candidates that lie in columns [c0, c1) from a copy of
// those columns (element j at src[j - c0]).
template <class In>
__device__ __forceinline__ void topk_gather(TopKLane& c, const void* src, int c0, int c1) {
  if (c.id0 >= c0 && c.id0 < c1) c.z0 = In::load1(src, c.id0 - c0);
  if (c.id1 >= c0 && c.id1 < c1) c.z1 = In::load1(src, c.id1 - c0);
}

// The parts of a row's CTAs (x = m, y = sw, z = acc), merged in rank order:
// the largest reference first, then every part rescaled to it (independent
// exponentials, no chain through the parts).
__device__ __forceinline__ TopKPart topk_merge_all(const float4* parts, int n) {
  float M = -INFINITY;
  for (int r = 0; r < n; ++r) M = fmaxf(M, parts[r].x);
  TopKPart p{M, 0.0f, 0.0f, 0};
  if (M == -INFINITY) return p;
  for (int r = 0; r < n; ++r) {
    const float4 e = parts[r];
    if (e.y > 0.0f) {
      const float f = ex2(e.x - M);
      p.sw = fmaf(f, e.y, p.sw);
      p.acc = fmaf(f, e.z, p.acc);
    }
  }
  return p;
}

// The warp's part over its lanes' candidates whose ids satisfy `mine`
// (fixed-order butterfly; every lane ends with it); k = log2(e) / T.
template <class Mine>
__device__ __forceinline__ TopKPart topk_part(const TopKLane& c, const TopKBuf* buf, int lane,
                                              float invT, float k, Mine mine) {
  const bool u0 = c.id0 >= 0 && mine(c.id0), u1 = c.id1 >= 0 && mine(c.id1);
  const int bad = __any_sync(0xffffffffu, c.bad) ? 1 : 0;
  const float t0 = c.z0 * k, t1 = c.z1 * k;
  float M = fmaxf(u0 ? t0 : -INFINITY, u1 ? t1 : -INFINITY);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  if (M == -INFINITY) return TopKPart{-INFINITY, 0.0f, 0.0f, bad};
  const float w0 = u0 ? ex2(t0 - M) : 0.0f, w1 = u1 ? ex2(t1 - M) : 0.0f;
  float sw = w0 + w1;
  float acc = (u0 ? w0 * fmaf(c.z0, invT, -buf->teacher[lane]) : 0.0f) +
              (u1 ? w1 * fmaf(c.z1, invT, -buf->teacher[lane + 32]) : 0.0f);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    sw += __shfl_xor_sync(0xffffffffu, sw, o);
    acc += __shfl_xor_sync(0xffffffffu, acc, o);
  }
  return TopKPart{M, sw, acc, bad};
}

// sw >= 1 (the largest candidate contributes 1), so a fast division is exact
// enough
__device__ __forceinline__ float topk_value(const TopKPart& p, float lse) {
  return p.sw > 0.0f ? __fdividef(p.acc, p.sw) - lse : 0.0f;
}

}  // namespace milesloss

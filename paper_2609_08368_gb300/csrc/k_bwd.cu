// dLogits from the per-row state a forward call saved (split forward /
// backward path): the logits are read once more, row statistics come from
// the workspace.
//   dZ_tj = g (m_t / N) (1/T) [G_t (1[j = y_t] - p_j) + gamma p_j (log p_j + H_t)]
// A tile is a contiguous run of kTile columns of one row; blocks stride
// over tiles. Each thread issues all of its 16-byte streaming loads of a tile
// (L1 skipped) before using any, then writes 16-byte streaming stores; rows
// that are not 16-byte aligned take the scalar path.
#include "common.cuh"
#include "kernels.h"

namespace milesloss {

namespace {

template <class In, class Out>
__global__ void __launch_bounds__(kBwdThreads) k_bwd(const BwdArgs a) {
  constexpr int V8 = In::kVec;
  using St = typename In::storage;
  WsPtrs ws = a.ws;
  const long long N = ws.hdr->n_tokens;
  float g = a.grad_loss;
  if (a.grad_loss_dev) g *= *a.grad_loss_dev;
  const float cscale = (N > 0) ? g / static_cast<float>(N) * a.invT : 0.0f;

  constexpr int kTile = kBwdTile;
  constexpr int kPer = kTile / V8 / kBwdThreads;  // vectors per thread per tile
  const bool vec = a.in_vec && a.out_vec;
  // Tile (row, t) of this block, advanced by gridDim.x tiles per step
  // without a division in the loop.
  const int tpr = a.tiles_per_row;
  const long long dq = gridDim.x / tpr;
  const int dr = static_cast<int>(gridDim.x % tpr);
  auto advance = [&](long long& row, int& t) {
    row += dq;
    t += dr;
    if (t >= tpr) { t -= tpr; ++row; }
  };
  // vectors of a tile (the last tile of a row may be partial; unaligned rows
  // take the scalar path)
  auto tile_nv = [&](int t) {
    const int j0 = t * kTile;
    return vec ? (min(a.V, j0 + kTile) - j0) / V8 : 0;
  };
  // All of a thread's 16-byte streaming loads of a tile are issued before
  // any is used, and the next tile's loads are issued before this tile's
  // arithmetic, so each thread keeps up to 2 kPer loads in flight.
  // rows that do not train (or have a bad target) get zeros: no read
  auto reads = [&](long long row) { return a.mask[row] != 0 && !(ws.flags[row] & kFlagBad); };
  auto load_tile = [&](long long row, int t, uint4* raw) {
    const int nv = reads(row) ? tile_nv(t) : 0;
    const char* zrow = static_cast<const char*>(a.logits) + row * a.ld * static_cast<long long>(sizeof(St)) +
                       static_cast<size_t>(t) * kTile * sizeof(St);
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int v = threadIdx.x + i * kBwdThreads;
      if (v < nv) raw[i] = ld_stream_u4(zrow + static_cast<size_t>(v) * 16);
    }
  };
  long long row = blockIdx.x / tpr;
  int t = static_cast<int>(blockIdx.x % tpr);
  uint4 raw[kPer], nxt[kPer];
  if (row < a.R) load_tile(row, t, raw);
  while (row < a.R) {
    long long nrow = row;
    int nt = t;
    advance(nrow, nt);
    if (nrow < a.R) load_tile(nrow, nt, nxt);
    const int j0 = t * kTile;
    const int j1 = min(a.V, j0 + kTile);
    const char* zrow = static_cast<const char*>(a.logits) + row * a.ld * static_cast<long long>(sizeof(St));
    char* drow = static_cast<char*>(a.dlogits) + row * a.ld_out * static_cast<long long>(Out::kSize);
    const int nv = tile_nv(t);
    const bool rd = reads(row);
    const float cc = rd ? cscale : 0.0f;
    const float G = ws.G[row], H = ws.H[row], lse = ws.lse[row];
    const float ca = cc * (-G + a.gamma * (H - lse));
    const float cb = cc * a.gamma * a.invT;
    const float L2 = lse * 1.4426950408889634f;
    // the target's column in this call's logits (outside [0, V): another
    // shard's, which no tile of this row holds)
    const int y = a.targets[row] - a.col0;
    const bool has_y = y >= j0 && y < j1;
    // The sampled token's entry (only in the tile that holds it):
    // cc [G (1 - p_y) + gamma p_y (log p_y + H)] with 1 - p_y = -expm1(logp),
    // accurate when p_y is close to 1.
    float dzy = 0.0f;
    if (has_y) {
      const float logp = ws.logp[row];
      dzy = cc * (G * -expm1f(logp) + a.gamma * expf(logp) * (logp + H));
    }
    auto value = [&](float z, int j) {
      if (j == y) return dzy;
      return (cc == 0.0f) ? 0.0f : ex2(fmaf(z, a.k, -L2)) * ent_factor(z, ca, cb);
    };
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int v = threadIdx.x + i * kBwdThreads;
      if (v >= nv) continue;
      const int jb = j0 + v * V8;
      float f[V8];
      if (cc == 0.0f) {  // (a row that does not train was not read)
#pragma unroll
        for (int e = 0; e < V8; ++e) f[e] = 0.0f;
      } else {
        In::unpack(raw[i], f);
#pragma unroll
        for (int e = 0; e < V8; ++e) f[e] = ex2(fmaf(f[e], a.k, -L2)) * ent_factor(f[e], ca, cb);
        if (has_y && static_cast<unsigned>(y - jb) < static_cast<unsigned>(V8)) {
#pragma unroll
          for (int e = 0; e < V8; ++e)
            if (jb + e == y) f[e] = dzy;
        }
      }
      Out::template storev<V8>(drow + static_cast<size_t>(jb) * Out::kSize, f, 0u);
    }
    for (int j = j0 + nv * V8 + threadIdx.x; j < j1; j += kBwdThreads)
      Out::store1(drow, j, cc == 0.0f ? 0.0f : value(In::load1(zrow, j), j));
#pragma unroll
    for (int i = 0; i < kPer; ++i) raw[i] = nxt[i];
    row = nrow;
    t = nt;
  }
}

}  // namespace

const void* bwd_kernel(rl_dtype in, rl_dtype out) {
  if (in == RL_BF16)
    return out == RL_BF16 ? reinterpret_cast<const void*>(&k_bwd<InBf16, OutBf16>)
                          : reinterpret_cast<const void*>(&k_bwd<InBf16, OutF32>);
  return out == RL_BF16 ? reinterpret_cast<const void*>(&k_bwd<InF32, OutBf16>)
                        : reinterpret_cast<const void*>(&k_bwd<InF32, OutF32>);
}

}  // namespace milesloss

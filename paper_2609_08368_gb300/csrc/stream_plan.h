// The streaming kernel's launch plan, in host-only C++ (no CUDA headers), so
// that the plan can be built and checked without a GPU: which rows k_stream
// takes, with how many CTAs per SM, and the shape of each CTA's ring of
// shared-memory slots. k_stream.cu reads the device's shared-memory limits
// and calls plan_ring; the host tests compile this header on its own.
#pragma once

#include <algorithm>

#include "milesloss.h"

namespace milesloss {

constexpr int kSweepSmemExtra = 1024;  // mbarriers + exchange + reduction scratch
constexpr int kMaxSlots = 16;          // ring slots of k_stream

// Which kernel sweeps rows of row_bytes, and with how many streaming CTAs per
// SM: 0 = the cluster kernel, 1 = one streaming CTA per SM (sixteen consumer
// warps, the whole shared memory for its ring), 2 or 4 = that many CTAs per SM
// (eight or four consumer warps, a half or a quarter of the shared memory),
// so that one CTA's per-row merge and epilogue overlap the other CTAs'
// passes. Rows must start 16-byte aligned to stream (else the cluster
// kernel). Measured on GB300 (fractions of the copy peak, A/B on one box,
// bf16 and fp32 rows):
//   fused: rows of 192-310 KB one CTA 0.966-0.984 against 0.939-0.959 in
//   clusters; 56-80 KB rows two CTAs 0.956-1.00 against 0.91-0.94; 20-56 KB
//   rows four CTAs 0.93-1.00 against 0.90-0.94 (48 KB fp32 rows: equal);
//   80-192 KB rows in clusters (0.93-0.99 by box; two CTAs ran from 2 % ahead
//   to 1 % behind on 96 KB rows, and one CTA with equal chunks from 3 % ahead
//   to 2 % behind on 136-184 KB bf16 rows, depending on the box), except fp32
//   rows of 120-136 KB (fp32_mid_row) and 136-192 KB (halves_row); 16 KB rows
//   in clusters (fp32 0.91 against 0.79 with four CTAs). With top-K OPD, four
//   CTAs per SM ran 6 % behind the clusters on 32 KB rows; two ran 3-4 %
//   ahead on 64 KB rows.
//   forward only: 200-310 KB rows one CTA (224 / 288 / 302 KB: 1.13 / 1.10
//   / 1.10 against 1.10 / 1.07 / 1.06 with two); 112-200 KB rows two CTAs
//   (151 KB: 1.05 against 0.94 with one, 192 KB: 1.08 against 1.06; a
//   read-only stream can pass the copy peak); 20-112 KB rows four CTAs
//   0.84-1.06 against 0.71-0.96 in clusters (64 KB fp32 rows: 1.07 against
//   1.08).
// The sweep_kernel override forces either kernel, stream_ctas_per_sm the
// CTAs per SM.

// fp32 rows of 120-136 KB (the fp32 workload's 32,768 columns), fused: two
// CTAs per SM with 18 KB chunks, 0.976 / 0.979 / 0.983 / 0.976 / 0.976
// against 0.970 / 0.960 / 0.969 / 0.968 / 0.962 in clusters on five boxes
// (bf16 rows of that length with those chunks: 0.87; with 24-36 KB chunks
// equal to the clusters).
inline bool fp32_mid_row(long long row_bytes, int es, bool grad, bool topk) {
  return grad && !topk && es == 4 && row_bytes > 120 * 1024 && row_bytes <= 136 * 1024;
}

// Fused fp32 rows of 136-192 KB: one CTA per SM with the row in two equal
// chunks (three ring slots up to 150 KB rows, two above), neither kept:
// against the clusters, rows of 136 / 144 / 152 / 160 / 176 KB ran +0.3 /
// +2.9 / +1.8 / +1.7 / +1.3 % on one box, 144 / 160 KB +4.1 / +3.5 % on
// another. (bf16 rows of that length: from 3 % ahead on one box to 2 % behind
// on another, where the clusters ran 0.96-0.99; they stay in clusters.)
inline bool halves_row(long long row_bytes, int es, bool grad) {
  constexpr long long KB = 1024;
  return grad && es == 4 && row_bytes >= 136 * KB && row_bytes < 192 * KB;
}

inline int stream_ctas(long long row_bytes, int es, bool grad, bool topk) {
  constexpr long long KB = 1024;
  if (grad) {
    if (row_bytes >= 192 * KB || halves_row(row_bytes, es, grad)) return 1;
    if (fp32_mid_row(row_bytes, es, grad, topk)) return 2;
    if (row_bytes > 56 * KB && row_bytes <= 80 * KB) return 2;
    if (!topk && row_bytes >= 20 * KB && row_bytes <= 56 * KB) return 4;
    return 0;
  }
  if (row_bytes >= 200 * KB) return 1;
  if (row_bytes > 112 * KB) return 2;
  if (row_bytes > 56 * KB) return topk ? 2 : 4;
  if (!topk && row_bytes >= 20 * KB) return 4;
  return 0;
}

// The ring. One CTA per SM, measured on GB300 among 44-112 KB chunks and 0-3
// kept chunks (bf16, fused): rows of 240 KB and more run best with three 74
// KB slots, the ragged remainder as the first chunk and the last two chunks
// kept for pass B (0.966-0.984 of the copy peak, against 0.959-0.973 with two
// 112 KB slots); shorter rows with two 112 KB slots and the last chunk kept
// (200 KB rows: 0.972-0.979, against 0.944 with 74 KB slots); a forward-only
// call has no pass B: two 112 KB slots. Several CTAs per SM, measured among
// 8-36 KB chunks and 1-3 kept chunks: two CTAs with three 36 KB slots (every
// chunk kept, up to three; six 18 KB slots for fp32_mid_row rows, three
// kept); four CTAs with the whole row in one slot up to 24 KB rows, else 16
// KB slots up to 44 KB rows, 12 KB slots up to 56 KB rows and 18 KB slots
// past that (forward only), the last chunk kept; chunks of 12 KB or less with
// two CTAs, or 8 KB with four, ran 10-45 % slower. The stream_* overrides
// force a chunk size, slot count, kept chunks, split and CTAs per SM.
constexpr long long kLongRowBytes = 240 * 1024;

struct SmemLimits {
  int optin;     // largest dynamic shared memory one CTA may opt in to
  int per_sm;    // shared memory of one SM
  int reserved;  // shared memory the system reserves per CTA
};

// The streaming kernel's launch plan (ring slots, kept chunks, split, shared
// memory per CTA, consumer warps, CTAs per row).
struct StreamPlan {
  int chunk, slots, hold, split_first, prefetch, smem;
  int cw;         // consumer warps per CTA: 16, 8 or 4 (one, two or four CTAs per SM)
  int cluster;    // CTAs per row: 1, or a cluster of 2, 4 or 8 (one CTA per SM)
  int slice_vec;  // with a cluster: whole 16-byte vectors of a row per CTA
};

// Fused calls without top-K: how many CTAs share a row (a thread-block
// cluster, each CTA streaming one slice of the row through its own ring, one
// CTA per SM). With one CTA per row and per SM, 152 rows are live at once and
// the second read of each row comes from L2 only while they fit in it; each
// row of a cluster costs one exchange between its CTAs, which short slices
// do not repay. Measured on
// GB300 (fractions of the copy peak, the glm recipe's rows with the
// vocabulary shown; one CTA / two / four per row):
//   bf16 400 KB 0.972 / 0.903, 448 KB 0.965 / 0.946, 512 KB 0.916 / 0.934 /
//   0.740, 1 MB - / 0.939 / 0.861, 1.5 MB - / 0.850 / 0.933, 2 MB 0.751 /
//   0.815 / 0.943 (eight: 0.724); fp32 400 KB 0.957 / 0.964, 620 KB 0.899 /
//   0.935 / 0.836; 310 KB (the glm rows) 0.978 / 0.831.
inline int stream_cluster(long long row_bytes, int es, bool grad, bool topk) {
  (void)es;
  constexpr long long KB = 1024;
  if (!grad || topk) return 1;
  if (row_bytes >= 1280 * KB) return 4;
  if (row_bytes >= 480 * KB) return 2;
  return 1;
}

// The whole 16-byte vectors of a row each CTA of a cluster of C takes: an
// even split rounded up to a multiple of 8 (every slice starts 128-byte
// aligned; the last CTA takes the rest, possibly nothing).
inline int slice_vectors(long long row_vec, int C) {
  return static_cast<int>(std::max(8LL, ((row_vec + C - 1) / C + 7) / 8 * 8));
}

// The plan for rows of row_bytes (elements of es bytes), given the SM's
// shared-memory limits, the extra shared memory beyond the ring and the
// fixed scratch (with top-K OPD on, its candidate buffers) and the
// overrides; false when a forced value does not fit.
inline bool plan_ring(long long row_bytes, int es, bool grad, bool topk, const SmemLimits& lim,
                      int extra, const rl_launch_overrides& ov, StreamPlan* out) {
  const int per = ov.stream_ctas_per_sm > 0 ? ov.stream_ctas_per_sm
                                            : std::max(1, stream_ctas(row_bytes, es, grad, topk));
  if (per != 1 && per != 2 && per != 4) return false;
  const bool lng = grad && row_bytes >= kLongRowBytes;
  const int budget = per > 1 ? std::min(lim.optin, lim.per_sm / per - lim.reserved) : lim.optin;
  int chunk_d = lng ? 75776 : 114688, hold_d = lng ? 2 : 1, split_d = lng ? 1 : 0;
  if (per == 1 && halves_row(row_bytes, es, grad)) {
    chunk_d = static_cast<int>(((row_bytes + 1) / 2 + 127) / 128 * 128);
    hold_d = 0;
    split_d = 1;
  } else if (per == 2) {
    chunk_d = fp32_mid_row(row_bytes, es, grad, topk) ? 18432 : 36864;
    hold_d = 3;
    split_d = 1;
  } else if (per == 4) {
    // (rows up to 56 KB take the same chunks in fused and forward-only
    // calls, so that both sum a row in the same order: the same bits)
    const long long whole = (row_bytes + 127) / 128 * 128;
    chunk_d = whole <= 24576 ? static_cast<int>(std::max(1024LL, whole))
                             : (row_bytes <= 44 * 1024 ? 16384
                                                       : (row_bytes <= 56 * 1024 ? 12288 : 18432));
    hold_d = 1;
    split_d = 1;
  }
  const int chunk = ov.stream_chunk_bytes > 0 ? ov.stream_chunk_bytes : chunk_d;
  if (chunk < 1024 || chunk > 131072 || chunk % 128) return false;
  int slots = (budget - kSweepSmemExtra - extra) / chunk;
  if (slots > kMaxSlots) slots = kMaxSlots;
  if (ov.stream_slots > 0) {
    if (ov.stream_slots > slots) return false;
    slots = ov.stream_slots;
  }
  if (slots < 1) return false;
  const int hold = ov.stream_hold >= 0 ? ov.stream_hold : std::min(hold_d, slots);
  if (hold > slots) return false;
  out->chunk = chunk;
  out->slots = slots;
  out->hold = hold;
  out->split_first = ov.stream_split_first >= 0 ? ov.stream_split_first : split_d;
  out->prefetch = ov.stream_prefetch_bytes >= 0 ? ov.stream_prefetch_bytes : 0;
  out->smem = slots * chunk + kSweepSmemExtra + extra;
  out->cw = 16 / per;
  out->cluster = 1;
  out->slice_vec = 0;
  return true;
}

// The plan with the row's CTAs: one (plan_ring over the whole row), or a
// cluster of C, whose CTAs each run plan_ring's one-CTA ring over their
// slice. Only fused calls without top-K run in clusters, and only when
// can_cluster (a call that writes the row's own results, not a vocabulary
// shard's records); other calls take one CTA per row whatever the
// stream_cluster override says, and so does a row whose CTAs per SM are
// forced above one (unless stream_cluster is forced too: no plan). False
// when a forced value does not fit.
inline bool plan_stream_rows(long long row_bytes, int es, bool grad, bool topk, bool can_cluster,
                             const SmemLimits& lim, int extra, const rl_launch_overrides& ov,
                             StreamPlan* out) {
  const bool can = can_cluster && grad && !topk;
  int C = 1;
  if (can && ov.stream_cluster > 0) C = ov.stream_cluster;
  else if (can && ov.stream_ctas_per_sm <= 1) C = stream_cluster(row_bytes, es, grad, topk);
  if (C == 1) return plan_ring(row_bytes, es, grad, topk, lim, extra, ov, out);
  if (C != 2 && C != 4 && C != 8) return false;
  if (ov.stream_ctas_per_sm > 1) return false;
  const int sv = slice_vectors(row_bytes / 16, C);
  rl_launch_overrides one = ov;
  one.stream_ctas_per_sm = 1;
  if (!plan_ring(static_cast<long long>(sv) * 16, es, grad, topk, lim, extra, one, out)) return false;
  out->cluster = C;
  out->slice_vec = sv;
  return true;
}

}  // namespace milesloss

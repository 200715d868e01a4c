// Internal interface between the C-ABI layer (abi.cu) and the kernels.
#pragma once

#include <cstdlib>

#include "common.cuh"
#include "stream_plan.h"

namespace milesloss {

constexpr int kMaxStages = 4;
constexpr int kMaxCluster = 8;
constexpr uint32_t kBulkChunk = 16384;    // bytes per cp.async.bulk
constexpr int kAdvThreads = 1024;
constexpr int kBwdThreads = 256;
// k_stream's block: cw consumer warps (16 with one CTA per SM, 8 with two, 4
// with four),
// the producer warp and, with top-K OPD, the top-K warp
constexpr int stream_threads(bool topk, int cw) { return cw * 32 + (topk ? 64 : 32); }
constexpr int kSeqThreads = 256;
constexpr int kAdvSmemBytes = 48 * 1024;  // on-chip trajectory tables when they fit
constexpr int kTopKSmem = 2 * (2 * kMaxTopK * 4);  // two rows of top-K ids + teacher values

struct SweepArgs {
  const void* logits;
  long long ld, R;
  int V;
  int slice;        // columns per CTA (multiple of 16 bytes of input)
  int stages;       // ring depth S
  int stage_bytes;  // bytes per stage (multiple of 128)
  int in_bulk;      // rows are 16-byte aligned: bulk-copy path
  int out_vec;      // dLogits rows are 16-byte aligned: vector stores
  const int* targets;
  const float* rho;
  const float* q;
  const float* old;
  const uint8_t* mask;
  float* out_logp;
  float* out_H;
  void* dlogits;
  long long ld_out;
  float grad_loss;
  const float* grad_loss_dev;
  LossScalars s;
  WsPtrs ws;
  // Test hook (0 = off): the first wait of every CTA waits instead on a
  // barrier nothing completes, bounded by this many nanoseconds, so that the
  // timeout path runs (see rl_launch_overrides).
  unsigned long long stall_ns;
  // A vocabulary-sharded call (forward only): the logits are columns
  // [col0, col0 + V) of a vocabulary of vocab_total ids, a target or top-K
  // candidate outside them is another shard's, and each row's partial sums
  // go to part_rows (two float4 per row, see k_vshard.cu) in place of the
  // epilogue. Unsharded calls: col0 0, vocab_total V, part_rows null.
  long long col0;
  int vocab_total;
  float4* part_rows;
};

struct StreamArgs {
  const void* logits;
  long long ld, R;
  int V;
  int chunk_bytes;  // bytes per ring slot (multiple of 128)
  int n_slots;      // ring depth
  int n_hold;       // last chunks of a row that pass B reads from shared memory (<= n_slots)
  int split_first;  // 1: the first chunk takes the ragged remainder (rounded up to 128 bytes)
  int prefetch;     // bytes of the next row to ask L2 for once a row's first pass is issued
  int out_vec;      // dLogits rows are 16-byte aligned: vector stores
  int slice_vec;    // launched in clusters (one per row): whole vectors of a row per CTA, a
                    // multiple of 8 (the cluster's last CTA may take fewer, or none)
  const int* targets;
  const float* rho;
  const float* q;
  const float* old;
  const uint8_t* mask;
  float* out_logp;
  float* out_H;
  void* dlogits;
  long long ld_out;
  float grad_loss;
  const float* grad_loss_dev;
  LossScalars s;
  WsPtrs ws;
  unsigned long long stall_ns;  // test hook, as in SweepArgs (the consumers' first wait)
  long long col0;               // vocabulary-sharded calls, as in SweepArgs
  int vocab_total;
  float4* part_rows;
};

struct AdvArgs {
  long long R;          // rows of this call (the local rows of a shard)
  long long row0;       // global index of local row 0 (0 unless sharded)
  long long R_total;    // rows of the whole call: cu_seqlens ends here (R unless sharded)
  const int* counts_in; // sharded calls: every trajectory's training tokens over all
                        // shards (then N and the per-trajectory counts come from these)
  int* counts_out;      // sharded calls: this shard's training tokens per trajectory
  int n_traj, n_groups;
  const float* rewards;
  const int* gid;
  const int* cu;
  const uint8_t* mask;
  const float* rho;
  const float* teacher;
  float opd_coef;
  int normalize_std, unbiased_std;
  float std_floor;
  int estimator;   // rl_estimator
  int smem_traj;   // trajectory tables (cu_seqlens, group ids, rewards, counts,
                   // advantages) staged in shared memory
  float* advantages;   // may be null
  int* group_sizes;    // may be null
  WsPtrs ws;
};

struct SeqArgs {
  const int* cu;        // row offsets of the whole call
  const float* rho;     // per-row arrays: this call's rows (local indices)
  const float* old;
  const float* q;
  const uint8_t* mask;
  long long row0, R;    // the call's rows are [row0, row0 + R) of the whole call
  // Sharded calls: sums_out receives, per trajectory, the sums over this
  // call's rows (sum of logp - base, sum of correction weights; [n_traj][2])
  // and nothing else is written; sums_in gives those sums added over every
  // shard, in place of the kernel's own.
  double* sums_out;
  const double* sums_in;
  LossScalars s;
  WsPtrs ws;
};

struct StatArgs {
  long long R;
  const uint8_t* mask;
  const float* rho;
  rl_loss_stats* out;
  rl_loss_partials* part_out;  // a shard: its partial sums instead of the statistics
  WsPtrs ws;
};

struct FinishArgs {
  const rl_loss_partials* part;
  rl_loss_stats* out;
};

struct BwdArgs {
  const void* logits;
  long long ld, R;
  int V;
  int tiles_per_row;
  long long n_tiles;
  int in_vec, out_vec;
  const int* targets;
  const uint8_t* mask;
  void* dlogits;
  long long ld_out;
  float grad_loss;
  const float* grad_loss_dev;
  float invT, k, gamma;
  int col0;  // the logits are columns [col0, col0 + V) of the vocabulary
  WsPtrs ws;
};

// The merge of a vocabulary-sharded call: each row's record from every
// column shard (two float4, shard-major: all[2 (k R + row)] and the one after
// it) in shard order, then the row's statistics and per-token objective, as
// the fused sweep's epilogue writes them.
constexpr int kMaxColShards = 64;
constexpr int kMergeThreads = 256;
struct MergeArgs {
  long long R;
  int n_shards;
  long long col_starts[kMaxColShards + 1];
  const float4* all;
  const int* targets;  // vocabulary ids
  const float* rho;
  const float* q;
  const float* old;
  const uint8_t* mask;
  float* out_logp;
  float* out_H;
  LossScalars s;
  WsPtrs ws;
};

constexpr int kBwdTile = kBwdThreads * 8 * 4;  // elements of one row per backward tile

// Kernel entry points (device function pointers usable with cudaLaunchKernelEx).
// topk: top-K OPD on (a separate instantiation, so that calls without it
// carry none of its code)
const void* sweep_kernel(rl_dtype in, rl_dtype out, bool grad, int threads, bool topk);
const void* sweep_kernel_topk(rl_dtype in, rl_dtype out, bool grad, int threads);
// clu: the instantiation that runs in clusters of CTAs per row (fused
// calls without top-K only; nullptr otherwise)
const void* stream_kernel(rl_dtype in, rl_dtype out, bool grad, bool topk, int cw, bool clu);

// The process-wide launch-plan overrides set by rl_set_launch_overrides (a
// copy; every field -1 when none are set).
rl_launch_overrides current_overrides();
// The status a workspace's error bits report: the lowest recorded code.
rl_status status_of_bits(uint32_t bits);

// The streaming kernel's launch plan (k_stream.cu, from the pure plan in
// stream_plan.h): whether rows of row_bytes go to it, and its ring of
// shared-memory slots.
bool use_stream(long long row_bytes, int es, bool in_bulk, bool grad, bool topk,
                const rl_launch_overrides& ov);
// extra: shared memory beyond the ring and the fixed scratch (kTopKSmem with
// top-K OPD on, else 0); the ring's shape depends on the row length and on
// whether the call writes dLogits
// (can_cluster: the call may run a row over a cluster of CTAs)
rl_status plan_stream(int dev, int extra, long long row_bytes, int es, bool grad, bool topk,
                      bool can_cluster, const rl_launch_overrides& ov, StreamPlan* out);
const void* bwd_kernel(rl_dtype in, rl_dtype out);
const void* adv_kernel();
const void* groups_kernel();  // one 32-thread block per group (grid-stride)
constexpr int kMaxGroupBlocks = 65535;
// Up to this many groups, k_advantages computes the group statistics itself
// (a launch costs more than their double arithmetic on one SM).
constexpr int kInlineGroups = 8;
const void* seq_kernel();
const void* merge_kernel();   // vocabulary-sharded calls: k_vmerge
const void* stats_kernel();
const void* finish_kernel();  // rl_loss_stats from combined partials (one thread)

}  // namespace milesloss

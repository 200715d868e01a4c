// rl_loss_fwd_bwd_noalloc: the fused forward+backward call for callers that
// cannot hand the library a device workspace.
//
// Some callers cannot allocate device memory when they call the loss:
// frameworks that reserve nearly all of HBM for their own pool at start-up
// (so a cudaMalloc from a library fails, or fragments and fights that
// pool), plain-C hosts and plugins that have no access to the process's
// allocator and so cannot size, own or free a buffer, and code paths whose
// memory footprint must stay fixed after initialisation. For them this
// entry point takes the same inputs and outputs as rl_loss_fwd_bwd but no
// workspace: the workspace is a fixed array compiled into the library.
//
// The array is kNoallocScratchBytes (8 MiB), enough for about 200,000 rows
// with small trajectory and group counts; every device on which the
// library's code is loaded keeps it until the process exits. Calls whose
// workspace would exceed it are rejected with RL_ERR_WORKSPACE_TOO_SMALL
// before anything is enqueued.
//
// Every call looks up the device address of the array on the current
// device (cudaGetSymbolAddress, with that device current). The address is
// not cached: after cudaDeviceReset, or in a new primary context, the
// library's device code is loaded again and the array may sit elsewhere.
// The first call on a device also loads that code, so make it before any
// stream capture. Nothing here calls cudaMalloc, cudaFree or any allocating
// routine.
//
// All calls on a device share the one array and it keeps the previous
// call's contents; the kernels reset what must start at zero (the error
// word and the reduction ticket) at the start of every call. Calls that
// overlap on the GPU (on different streams, or from different host
// threads) race on the array and must be serialised by the caller. The
// data-dependent error word stays in the array after a call:
// rl_loss_noalloc_check_device_error reads it back (cudaMemcpyFromSymbol,
// no allocation); rows with a bad target get zeros as in rl_loss_fwd_bwd.
#include <cuda_runtime.h>

#include "kernels.h"
#include "milesloss.h"

namespace {

constexpr size_t kNoallocScratchBytes = size_t(8) << 20;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

// Device address of the scratch array on the current device.
rl_status scratch_address(void** out) {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return RL_ERR_CUDA;
  *out = p;
  return RL_OK;
}

}  // namespace

extern "C" rl_status rl_loss_fwd_bwd_noalloc(
    const void* logits, rl_dtype logits_dtype, int64_t n_rows, int64_t vocab, int64_t ld,
    const int32_t* targets, const float* rollout_logprobs, const float* ref_logprobs,
    const float* old_logprobs, const float* teacher_logprobs, const float* rewards,
    const int32_t* group_id, const int32_t* cu_seqlens, int32_t n_traj, int32_t n_groups,
    const uint8_t* loss_mask, const rl_loss_params* params, float* token_logprobs,
    float* entropy, float* advantages, int32_t* group_sizes, rl_loss_stats* stats,
    float grad_loss, const float* grad_loss_device, void* dlogits, rl_dtype dlogits_dtype,
    int64_t ld_out, rl_stream stream) {
  size_t need = 0;
  rl_status st = rl_loss_workspace_size(n_rows, n_traj, n_groups, &need);
  if (st != RL_OK) return st;
  if (need > kNoallocScratchBytes) return RL_ERR_WORKSPACE_TOO_SMALL;
  void* scratch = nullptr;
  st = scratch_address(&scratch);
  if (st != RL_OK) return st;
  return rl_loss_fwd_bwd(logits, logits_dtype, n_rows, vocab, ld, targets, rollout_logprobs,
                         ref_logprobs, old_logprobs, teacher_logprobs, rewards, group_id,
                         cu_seqlens, n_traj, n_groups, loss_mask, params, token_logprobs,
                         entropy, advantages, group_sizes, stats, grad_loss, grad_loss_device,
                         dlogits, dlogits_dtype, ld_out, scratch, kNoallocScratchBytes, stream);
}

extern "C" rl_status rl_loss_noalloc_check_device_error(void) {
  // The error word is the first field of the workspace header, which starts
  // the array (milesloss::WsLayout puts the header at offset 0).
  uint32_t bits = 0;
  if (cudaMemcpyFromSymbol(&bits, g_noalloc_scratch, sizeof(bits), 0, cudaMemcpyDeviceToHost) !=
      cudaSuccess)
    return RL_ERR_CUDA;
  return milesloss::status_of_bits(bits);
}

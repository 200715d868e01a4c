// The cluster kernel's instantiations with top-K OPD (Sec. 5.2) on.
#include "k_sweep.cuh"

namespace milesloss {

namespace {

template <class In, class Out, bool kGrad>
const void* pick_topk(int threads) {
  switch (threads) {
    case 256: return reinterpret_cast<const void*>(&k_sweep<In, Out, kGrad, 256, 4, true>);
    case 255: return reinterpret_cast<const void*>(&k_sweep<In, Out, kGrad, 256, 5, true>);  // 5 per SM
    default: return reinterpret_cast<const void*>(&k_sweep<In, Out, kGrad, 512, 2, true>);
  }
}

}  // namespace

const void* sweep_kernel_topk(rl_dtype in, rl_dtype out, bool grad, int threads) {
  if (!grad) return in == RL_BF16 ? pick_topk<InBf16, OutBf16, false>(threads)
                                  : pick_topk<InF32, OutF32, false>(threads);
  if (in == RL_BF16) return out == RL_BF16 ? pick_topk<InBf16, OutBf16, true>(threads)
                                           : pick_topk<InBf16, OutF32, true>(threads);
  return out == RL_BF16 ? pick_topk<InF32, OutBf16, true>(threads)
                        : pick_topk<InF32, OutF32, true>(threads);
}

}  // namespace milesloss

// The cluster kernel's instantiations without top-K OPD; those with it are
// compiled in k_sweep_topk.cu (a translation unit of their own, built in
// parallel).
#include "k_sweep.cuh"

namespace milesloss {

namespace {

template <class In, class Out, bool kGrad>
const void* pick(int threads) {
  switch (threads) {
    case 256: return reinterpret_cast<const void*>(&k_sweep<In, Out, kGrad, 256, 4, false>);
    case 255: return reinterpret_cast<const void*>(&k_sweep<In, Out, kGrad, 256, 5, false>);  // 5 per SM
    default: return reinterpret_cast<const void*>(&k_sweep<In, Out, kGrad, 512, 2, false>);
  }
}

}  // namespace

const void* sweep_kernel(rl_dtype in, rl_dtype out, bool grad, int threads, bool topk) {
  if (topk) return sweep_kernel_topk(in, out, grad, threads);
  if (!grad) return in == RL_BF16 ? pick<InBf16, OutBf16, false>(threads)
                                  : pick<InF32, OutF32, false>(threads);
  if (in == RL_BF16) return out == RL_BF16 ? pick<InBf16, OutBf16, true>(threads)
                                           : pick<InBf16, OutF32, true>(threads);
  return out == RL_BF16 ? pick<InF32, OutBf16, true>(threads) : pick<InF32, OutF32, true>(threads);
}

}  // namespace milesloss

// Prints the streaming kernel's launch plan (stream_plan.h, host-only) for a
// grid of row lengths, element sizes, fused / forward-only calls and top-K on
// or off, for the limits of one GB300 SM (227 KB of shared memory a CTA may
// opt in to, 228 KB per SM, 1 KB reserved per CTA). One line per case:
//   es grad topk row_bytes ctas ok chunk slots hold split smem cw cluster slice_vec
// (rows of 1 to 320 KB in steps of 1 KB, then to 4 MB in steps of 32 KB)
#include <cstdio>

#include "stream_plan.h"

int main(int argc, char** argv) {
  using namespace milesloss;
  const SmemLimits lim{232448, 233472, 1024};
  rl_launch_overrides none;
  none.sweep_kernel = none.cluster_size = none.cluster_stages = none.cluster_threads = -1;
  none.cluster_ctas_per_sm = none.stream_chunk_bytes = none.stream_slots = none.stream_hold = -1;
  none.stream_split_first = none.stream_prefetch_bytes = none.stream_ctas_per_sm = -1;
  none.stall_first_wait_ns = -1;
  none.stream_cluster = -1;
  if (argc > 1) {
    // forced plans of a fused bf16 row of 512 KB: "per clu topk" per line,
    // printed as "ok cluster cw"
    const int cases[][3] = {{-1, -1, 0}, {2, -1, 0}, {4, -1, 0}, {1, -1, 0}, {-1, 4, 0},
                            {1, 8, 0}, {2, 2, 0}, {-1, 4, 1}, {-1, 1, 0}};
    for (const auto& c : cases) {
      rl_launch_overrides o = none;
      o.stream_ctas_per_sm = c[0];
      o.stream_cluster = c[1];
      StreamPlan p{};
      const bool ok = plan_stream_rows(512 * 1024, 2, true, c[2] != 0, true, lim,
                                       c[2] ? 1024 : 0, o, &p);
      std::printf("%d %d %d %d %d %d\n", c[0], c[1], c[2], ok ? 1 : 0, ok ? p.cluster : 0,
                  ok ? p.cw : 0);
    }
    return 0;
  }
  for (int es = 2; es <= 4; es += 2)
    for (int grad = 0; grad <= 1; ++grad)
      for (int topk = 0; topk <= 1; ++topk)
        for (long long kb = 1; kb <= 4096; kb += (kb < 320 ? 1 : 32))
          for (int d = -16; d <= 16; d += 16) {
            const long long row = kb * 1024 + d;
            StreamPlan p{};
            const int ctas = stream_ctas(row, es, grad, topk);
            const bool ok =
                plan_stream_rows(row, es, grad, topk, true, lim, topk ? 1024 : 0, none, &p);
            std::printf("%d %d %d %lld %d %d %d %d %d %d %d %d %d %d\n", es, grad, topk, row, ctas,
                        ok ? 1 : 0, p.chunk, p.slots, p.hold, p.split_first, p.smem, p.cw,
                        p.cluster, p.slice_vec);
          }
  return 0;
}

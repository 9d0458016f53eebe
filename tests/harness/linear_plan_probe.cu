// Host-side probe of the SM-pair perturbed-linear planner (zo_linear_pair.cu): prints, for a
// grid of shapes, ranks and pair counts, the automatic tiling and every pair tiling's plan,
// one line each:
//   T m n r n_pairs tiling N pairs group n_contrib s_cols s_split s_chunk auto
// Built and run by tests/test_linear_plan_cpu.py, which checks each plan's invariants and
// that its tile order completes.  Calls no CUDA function.
#include <cstdio>

#include "zo_kernels.h"

int main() {
  const long long Ts[] = {1, 130, 256, 300, 2000, 4096, 8192, 19500};
  const long long ms[] = {64, 136, 304, 1032, 4096, 11008};
  const long long ns[] = {72, 520, 4096, 11008};
  const int rs[] = {16, 32, 64, 128};
  const int pairs[] = {1, 2, 3, 5, 37, 74, 76};
  for (long long T : Ts)
    for (long long m : ms)
      for (long long n : ns)
        for (int r : rs)
          for (int np : pairs) {
            const int a = zo::linear_pair_tiling(T, m, n, r, np);
            for (int t = zo::kLinearPairTiling0; t < zo::kLinearPairTiling0 + 5; ++t) {
              const zo::LinearPairPlan p = zo::linear_pair_plan(T, m, n, r, t, np);
              std::printf("%lld %lld %lld %d %d %d %d %d %d %d %d %d %d %d\n", T, m, n, r, np, t,
                          zo::linear_pair_cols(t), p.pairs, p.group, p.n_contrib, p.s_cols,
                          p.s_split, p.s_chunk, a);
            }
          }
  return 0;
}

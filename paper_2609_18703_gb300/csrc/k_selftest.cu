// k_selftest.cu — a self-test of the bounded device-side waits.
//
// Every wait of the lineage kernels (a decoupled look-back on a predecessor
// tile, the one-pass admission's grid barrier, the copy's stage barriers) is
// bounded: past SPIN_LIMIT polls it records ERR_TIMEOUT in the context and
// returns, so that the context stays usable and the host reports
// RO_E_TIMEOUT.  This kernel runs one such wait that nothing releases, on
// scratch state of its own:
//   kind 0  a look-back of tile 1 whose predecessor never publishes;
//   kind 1  a grid barrier of two CTAs of which one never arrives.
#include "ro_internal.h"

namespace ro {

__global__ void __launch_bounds__(32) selftest_wait_kernel(SelftestArgs a) {
  if (a.kind == 0) {
    lookback_exclusive(a.ts, 1u, 1ull, a.epoch, a.err);
  } else if (blockIdx.x == 0) {
    grid_barrier(a.rs, 1u, a.err);   // CTA 1 returns without arriving
  }
}

void launch_selftest(cudaStream_t s, const SelftestArgs& a) {
  selftest_wait_kernel<<<a.kind == 0 ? 1 : 2, 32, 0, s>>>(a);
}

}  // namespace ro

// Checks by region, step 3, the variant with the open column's rows in shared
// memory, and its launcher.
#include <cuda_runtime.h>

#include "launch.h"
#include "region_check.cuh"

namespace epic {

void launch_check_sm(dim3 grid, dim3 block, size_t dyn, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
        const int32_t* x, int n, const int32_t* pos, int k, const int32_t* cand, int K, long long total,
        uint8_t* valid, const SeqPack& sp, const WPack& wp, int32_t* regs, int rmax, unsigned long long* counter,
        unsigned long long* stats) {
  cudaFuncSetAttribute(k_check<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  k_check<true><<<grid, block, dyn, st>>>(g, table, vocab, x, n, pos, k, cand, K, total, valid, sp, wp, regs, rmax,
                                        counter, stats);
}

// measurement builds: this translation unit's phase counters of the walk
int phase_read_check_sm(unsigned long long* out16, int reset) {
#ifdef EPIC_PHASE_TIMERS
  unsigned long long h[16];
  if (cudaMemcpyFromSymbol(h, g_phase, sizeof(h)) != cudaSuccess) return -1;
  for (int i = 0; i < 16; ++i) out16[i] += h[i];
  if (reset) {
    unsigned long long z[16] = {0};
    if (cudaMemcpyToSymbol(g_phase, z, sizeof(z)) != cudaSuccess) return -1;
  }
#else
  (void)out16;
  (void)reset;
#endif
  return 0;
}

}  // namespace epic

// Whole-graph walks: one warp per validity check (kernel and launcher).
#include <cuda_runtime.h>

#include "launch.h"

using namespace epic;

// K2-K4 (warp form): one warp per validity check; warps pull checks from a
// counter.  Each check walks the lexeme graph of x (+) (pos, tok) and runs
// bit-parallel Earley recognition over it.
// Copy the walk's grammar tables into shared memory and point `out` at them.
__device__ void stage_grammar(const DevGrammar& g, unsigned char* smem, DevGrammar& out) {
  out = g;
  unsigned char* p = smem;
  auto put = [&](const void* src, size_t bytes) -> void* {
    void* dst = p;
    const uint32_t* s4 = (const uint32_t*)src;
    uint32_t* d4 = (uint32_t*)dst;
    size_t n4 = bytes / 4;
    for (size_t i = threadIdx.x; i < n4; i += blockDim.x) d4[i] = s4[i];
    for (size_t i = n4 * 4 + threadIdx.x; i < bytes; i += blockDim.x)
      ((unsigned char*)dst)[i] = ((const unsigned char*)src)[i];
    p += (bytes + 15) & ~(size_t)15;
    return dst;
  };
  out.exp_term = (const uint32_t*)put(g.exp_term, (size_t)g.T * g.W * 4);
  out.exp_nt = (const uint32_t*)put(g.exp_nt, (size_t)g.V * g.W * 4);
  out.pred = (const uint32_t*)put(g.pred, (size_t)g.V * g.W * 4);
  out.gap_pred = (const uint32_t*)put(g.gap_pred, (size_t)g.V * g.W * 4);
  out.any_nt = (const uint32_t*)put(g.any_nt, (size_t)g.W * 4);
  out.any_term = (const uint32_t*)put(g.any_term, (size_t)g.W * 4);
  out.next_any = (const uint32_t*)put(g.next_any, (size_t)g.W * 4);
  out.nullable_next = (const uint32_t*)put(g.nullable_next, (size_t)g.W * 4);
  out.complete = (const uint32_t*)put(g.complete, (size_t)g.W * 4);
  out.item_next = (const int16_t*)put(g.item_next, (size_t)g.D * 2);
  out.item_lhs = (const int16_t*)put(g.item_lhs, (size_t)g.D * 2);
  out.dfa_accept = (const int16_t*)put(g.dfa_accept, (size_t)g.Q * 2);
  out.dfa_ext = (const uint8_t*)put(g.dfa_ext, (size_t)g.Q);
  out.skip = (const uint8_t*)put(g.skip, (size_t)g.T);
  __syncthreads();
}

template <bool SM>
__global__ void __launch_bounds__(32 * kWarpsPerCta) k_validate_warp(
    DevGrammar g, const LexEntry* __restrict__ table, int vocab, const int32_t* __restrict__ x, int n,
    const int32_t* __restrict__ pos, int k, const int32_t* __restrict__ cand, int K, long long total,
    uint8_t* __restrict__ valid, WPack wp, int rmax, int gtab_smem, unsigned long long* counter,
    unsigned long long* stats) {
  __shared__ WSh shm[kWarpsPerCta];
  extern __shared__ __align__(16) unsigned char dyn[];
  int warp = threadIdx.x >> 5;
  WSh& sh = shm[warp];
  for (int w = threadIdx.x & 31; w < kWCols / 32; w += 32) {
    sh.touched[w] = 0;
    sh.dirty[w] = 0;
  }
  for (int v = threadIdx.x & 31; v < kWMaxVW; v += 32) {
    sh.vset[v] = 0;
    sh.vdone[v] = 0;
  }
  __syncwarp();
  // the grammar tables in shared memory when they fit (gtab > 0)
  DevGrammar gs = g;
  size_t gt = 0;
  if constexpr (SM) {
    if (gtab_smem) {
      stage_grammar(g, dyn, gs);
      gt = gtab_bytes(g.T, g.V, g.W, g.D, g.Q);
    }
  }
  WarpWalker<SM> walk(gs, table, wp.carve((long long)blockIdx.x * (blockDim.x >> 5) + warp), sh, wp.nmax, wp.emax,
                      vocab);
  if constexpr (SM) {
    size_t per = smem_per_warp(wp.nmax, rmax, g.W, g.VW);
    unsigned char* base = dyn + gt + per * warp;
    uint32_t* rows = (uint32_t*)base;
    uint32_t* bd = rows + (size_t)rmax * g.W;
    int32_t* sorg = (int32_t*)(bd + (size_t)rmax * g.VW);
    uint32_t* ssum = (uint32_t*)(sorg + rmax);
    int16_t* so = (int16_t*)(ssum + 2 * rmax);
    walk.set_smem(rows, bd, so, sorg, ssum, rmax);
  }
  unsigned long long n_checks = 0, n_valid = 0, n_ovf = 0, n_bad = 0, n_cols = 0, n_ent = 0;
  for (;;) {
    long long jb = 0;
    if ((threadIdx.x & 31) == 0) jb = (long long)atomicAdd(counter, 1ull);
    jb = __shfl_sync(0xffffffffu, jb, 0);
    if (jb >= total) break;
    long long b = jb / ((long long)k * K);
    long long j = (jb / K) % k;
    int r = walk.run(x + b * n, n, pos[b * k + j], cand[jb]);
    if ((threadIdx.x & 31) == 0) valid[jb] = r == 1 ? 1 : (r == -1 ? 2 : 0);
    ++n_checks;
    n_valid += r == 1;
    n_ovf += r == -1;
    n_bad += r == -2;
    n_cols += walk.ncols;
    n_ent += walk.nent;
  }
  if ((threadIdx.x & 31) == 0 && n_checks) {
    atomicAdd(&stats[S_CHECKS], n_checks);
    atomicAdd(&stats[S_VALID], n_valid);
    atomicAdd(&stats[S_OVERFLOW], n_ovf);
    atomicAdd(&stats[S_BAD], n_bad);
    atomicAdd(&stats[S_COLUMNS], n_cols);
    atomicAdd(&stats[S_ENTRIES], n_ent);
  }
}


namespace epic {

void launch_validate_warp(bool sm, dim3 grid, dim3 block, size_t dyn, cudaStream_t st, const DevGrammar& g,
                          const LexEntry* table, int vocab, const int32_t* x, int n, const int32_t* pos, int k,
                          const int32_t* cand, int K, long long total, uint8_t* valid, const WPack& wp, int rmax,
                          int gsm, unsigned long long* counter, unsigned long long* stats) {
  if (sm) {
    cudaFuncSetAttribute(k_validate_warp<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
    k_validate_warp<true><<<grid, block, dyn, st>>>(g, table, vocab, x, n, pos, k, cand, K, total, valid, wp, rmax,
                                                    gsm, counter, stats);
  } else {
    k_validate_warp<false><<<grid, block, dyn, st>>>(g, table, vocab, x, n, pos, k, cand, K, total, valid, wp, rmax,
                                                     gsm, counter, stats);
  }
}

int phase_read_walk(unsigned long long* out16, int reset) {
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

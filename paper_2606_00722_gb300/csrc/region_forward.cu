// Checks by region, step 1: the forward chart of x per sequence (warp walk
// or block walk, both recording the graph), with its launchers.
#include <cuda_runtime.h>

#include "launch.h"
#include "region.cuh"

namespace epic {

// ------------------------------------------------------------------ 1. forward chart
template <bool SM>
__global__ void __launch_bounds__(32 * kWarpsPerCta) k_forward(DevGrammar g, const LexEntry* __restrict__ table,
                                                                int vocab, const int32_t* __restrict__ x, int B, int n,
                                                                SeqPack sp, int rmax,
                                                                unsigned long long* stats) {
  __shared__ WSh shm[kWarpsPerCta];
  extern __shared__ __align__(16) unsigned char dyn[];
  int warp = threadIdx.x >> 5;
  long long b = (long long)blockIdx.x * (blockDim.x >> 5) + warp;
  if (b >= B) return;
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
  SeqArena a = sp.carve(b);
  // the walk expects a zeroed stage and completion record
  for (size_t w = threadIdx.x & 31; w < (size_t)sp.nmax * g.W; w += 32) a.ws.stage[w] = 0;
  for (size_t w = threadIdx.x & 31; w < (size_t)sp.nmax * g.VW; w += 32) a.ws.bdone[w] = 0;
  __syncwarp();
  WarpWalker<SM, true> walk(g, table, a.ws, sh, sp.nmax, sp.emax, vocab);
  if constexpr (SM) {
    size_t per = smem_per_warp(sp.nmax, rmax, g.W, g.VW);
    unsigned char* base = dyn + per * warp;
    uint32_t* rows = (uint32_t*)base;
    uint32_t* bd = rows + (size_t)rmax * g.W;
    int32_t* sorg = (int32_t*)(bd + (size_t)rmax * g.VW);
    uint32_t* ssum = (uint32_t*)(sorg + rmax);
    int16_t* so = (int16_t*)(ssum + 2 * rmax);
    walk.set_smem(rows, bd, so, sorg, ssum, rmax);
  }
  SeqRec rec = a.rec;
  walk.rec = &rec;
  for (int p = threadIdx.x & 31; p < n; p += 32) {
    rec.gap_col[p] = -1;
    rec.pre_col[p] = -1;
    rec.post_col[p] = -1;
  }
  __syncwarp();
  int r = walk.run(x + b * n, n, -1, 0);
  if ((threadIdx.x & 31) == 0) {
    rec.meta[M_NCOLS] = walk.ncols;
    rec.meta[M_NEDGES] = rec.n_edges;
    rec.meta[M_START] = walk.start_col;
    rec.meta[M_STATUS] = r == 1 ? 1 : (r == 0 ? 0 : -1);
    rec.meta[M_NENT] = (int)walk.nent;
    atomicAdd(&stats[4], (unsigned long long)walk.ncols);  // columns and entries of the forward charts
    atomicAdd(&stats[5], (unsigned long long)walk.nent);
  }
}

// The same forward charts with a whole CTA per sequence (wide grammars,
// long rows): the Gauss-Seidel column closure of gscols.cuh, the CTA
// scattering each origin's completions.  The grammar's per-item tables sit in
// dynamic shared memory.
__global__ void __launch_bounds__(32 * kGsMaxWarps, 1) k_forward_gs(DevGrammar g, const LexEntry* __restrict__ table,
                                                                    int vocab, const int32_t* __restrict__ x, int B,
                                                                    int n, SeqPack sp, unsigned long long* stats) {
  __shared__ WalkShared sh;
  __shared__ GsShared gss;
  extern __shared__ __align__(16) unsigned char dyn[];
  GsTables tb;
  gs_stage_tables(g, dyn, tb);
  for (long long b = blockIdx.x; b < B; b += gridDim.x) {
    SeqArena a = sp.carve(b);
    // the walk expects a zeroed stage and completion record
    for (size_t w = threadIdx.x; w < (size_t)sp.nmax * g.W; w += blockDim.x) a.ws.stage[w] = 0;
    for (size_t w = threadIdx.x; w < (size_t)sp.nmax * g.VW; w += blockDim.x) a.ws.bdone[w] = 0;
    for (int p = threadIdx.x; p < n; p += blockDim.x) {
      a.rec.gap_col[p] = -1;
      a.rec.pre_col[p] = -1;
      a.rec.post_col[p] = -1;
    }
    __syncthreads();
    Workspace ws;
    ws.stage = a.ws.stage;
    ws.bdone = a.ws.bdone;
    ws.col_off = a.ws.col_off;
    ws.org = a.ws.org;
    ws.bits = a.ws.bits;
    ws.cov = nullptr;
    WalkScratch sc;
    sc.g_src = a.ws.g_src;
    sc.g_end = a.ws.g_end;
    sc.g_len = a.ws.g_len;
    sc.g_tail = (uint8_t*)a.ws.g_tail;  // [kMaxQ][16] bytes
    sc.g_lbl = a.ws.g_lbl;
    sc.g_last = a.ws.g_last;
    sc.f_q = a.ws.f_q;
    sc.f_c = a.ws.f_c;
    sc.key_q = a.key_q;
    sc.expn = nullptr;
    sc.bnew = nullptr;
    const BlockRec br{a.rec.col_gap, a.rec.e_dst,   a.rec.e_src,   a.rec.e_lbl,    a.rec.cnt,
                      a.ws.esum,     a.rec.gap_col, a.rec.pre_col, a.rec.post_col, a.rec.edge_cap};
    WsDims d;
    d.nmax = sp.nmax;
    d.emax = sp.emax;
    EarleyColsGS<true> cols(g, tb, table, ws, sc, d, sh, gss);
    cols.rec = &br;
    cols.wnt = (uint32_t*)(dyn + gs_tables_bytes(g.D, g.W, g.adv_steps));
    cols.wscr = cols.wnt + (size_t)kGsMaxWarps * kMaxVW;
    cols.par = g.gs_par != 0;
    Walk<EarleyColsGS<true>> walk(cols, g, table, sc, sh, vocab);
    walk.rec = &br;
    Subst none{nullptr, nullptr, 0};
    const int r = walk.run(x + b * n, n, none);
    __syncthreads();
    if (threadIdx.x == 0) {
      int32_t* meta = a.rec.meta;
      meta[M_NCOLS] = sh.ncols;
      meta[M_NEDGES] = sh.nedges;
      meta[M_START] = sh.start_col;
      meta[M_ACCEPT] = sh.accept_col;
      meta[M_STATUS] = r == 1 ? 1 : (r == 0 ? 0 : -1);
      meta[M_NENT] = (int)sh.nent;
      atomicAdd(&stats[4], (unsigned long long)sh.ncols);
      atomicAdd(&stats[5], (unsigned long long)sh.nent);
    }
    __syncthreads();
  }
}

void launch_forward(bool sm, dim3 grid, dim3 block, size_t dyn, cudaStream_t st, const DevGrammar& g,
                    const LexEntry* table, int vocab, const int32_t* x, int B, int n, const SeqPack& sp, int rmax,
                    unsigned long long* stats) {
  if (sm) {
    cudaFuncSetAttribute(k_forward<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
    k_forward<true><<<grid, block, dyn, st>>>(g, table, vocab, x, B, n, sp, rmax, stats);
  } else {
    k_forward<false><<<grid, block, dyn, st>>>(g, table, vocab, x, B, n, sp, rmax, stats);
  }
}

void launch_forward_gs(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
                       const int32_t* x, int B, int n, const SeqPack& sp, unsigned long long* stats) {
  const size_t dyn =
      gs_tables_bytes(g.D, g.W, g.adv_steps) + (size_t)kGsMaxWarps * kMaxVW * 4 + gs_warp_scratch_bytes();
  DevGrammar gg = g;
  gg.gs_par = gs_parallel_enabled(g.W);
  cudaFuncSetAttribute(k_forward_gs, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  k_forward_gs<<<grid, 32 * kGsMaxWarps, dyn, st>>>(gg, table, vocab, x, B, n, sp, stats);
}

// measurement builds: this translation unit's phase counters of the walk
int phase_read_forward(unsigned long long* out16, int reset) {
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

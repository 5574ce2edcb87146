// Validity checks by region, for grammars whose charts are large.
//
// Every check x (+) (i, t) differs from x only around position i.  So:
//  1. k_forward: one forward chart F of x per sequence (one warp each),
//     recording its graph (edges, gap flags), where each position's segment
//     sits in it, and each entry's completed nonterminals.  If x itself is
//     not completable, no single update is (the update's completion language
//     is a subset of x's), and every check of the sequence is 0.
//  2. k_good: a backward pass over F marks the "good" items: an item
//     (p, d, o) at node j is good if its own closure -- scanning along the
//     graph after j, nested constituents completing where F records them,
//     and its completion advancing the items waiting at column o -- reaches
//     the accepting item.  Such a closure uses only the graph after j and
//     the columns at o and before, so it is the same in every check whose
//     region lies after o and before j.
//  3. k_check: per check, only the region is walked (the candidate's span,
//     merged with fixed neighbours) with lookbacks into F; from the first
//     node after the region on, an item whose origin is an F node is
//     resolved by its good mask, and only the items whose origin lies in the
//     region are carried forward over F's graph.  The check is valid iff a
//     good item is found (or the accepting item, when the region holds the
//     start or the end).
#pragma once
#include "warpwalk.cuh"

namespace epic {

// Per-sequence forward chart and its tables.
struct SeqArena {
  WWs ws;          // the forward walk's workspace; org/bits/esum/col_off are the chart
  SeqRec rec;
  uint32_t* good;      // [emax][W]
  int32_t* last_col;   // [nmax] last column holding origin u (-1: none)
  int32_t* in_off;     // [nmax + 1] edges are stored by target column
  int32_t* out_off;    // [nmax + 1]
  int32_t* out_idx;    // [edge_cap]
  int32_t* succ_off;   // [nmax + 1] columns holding origin u, ascending
  int32_t* succ_idx;   // [emax]
  uint32_t* expn;      // [nmax][W] scratch of the good pass
  int32_t* eidx;       // [nmax (nmax + 1) / 2] entry of (column j, origin o <= j), -1: none
  uint8_t* gnz;        // [emax] the entry has a good item
  int32_t* cursor;     // [2 (nmax + 1)] scratch of the good pass
  int32_t* key_q;      // [kMaxQ] scratch of the block forward walk
  uint32_t* bexpn;     // [nmax][W]
  uint32_t* bnew;      // [nmax][VW]
};

struct SeqPack {
  char* base;
  size_t per_seq;
  int nmax, n, W, VW, edge_cap;
  long long emax;
  __host__ __device__ static size_t r(size_t b) { return (b + 255) & ~(size_t)255; }
  __host__ __device__ size_t bytes() const {
    size_t nm = nmax;
    return r(nm * W * 4) + r(nm * VW * 4) + r((nm + 1) * 4) + 6 * r(kWMaxQ * 4) + r(kWMaxQ * 16) + r(kWMaxQ * 32) +
           r(nm * 8) + r((size_t)emax * 4) + r((size_t)emax * 8) + r((size_t)emax * W * 4)  // WWs
           + r(nm) + 2 * r((size_t)edge_cap * 4) + r((size_t)edge_cap * 32) + 3 * r((size_t)n * 4) +
           r((size_t)emax * VW * 4) + r(32)                                                 // SeqRec
           + r((size_t)emax * W * 4) + r(nm * 4) + 3 * r((nm + 1) * 4) + r((size_t)edge_cap * 4) +
           r((size_t)emax * 4) + r(nm * W * 4) + r(nm * (nm + 1) / 2 * 4) + r((size_t)emax) + r(2 * (nm + 1) * 4) + r(kMaxQ * 4) +
           r(nm * W * 4) + r(nm * VW * 4);
  }
  __device__ SeqArena carve(long long b) const {
    SeqArena a;
    char* p = base + per_seq * (size_t)b;
    auto take = [&](size_t bytes) {
      char* q = p;
      p += r(bytes);
      return q;
    };
    size_t nm = nmax;
    a.ws.stage = (uint32_t*)take(nm * W * 4);
    a.ws.bdone = (uint32_t*)take(nm * VW * 4);
    a.ws.col_off = (int32_t*)take((nm + 1) * 4);
    a.ws.f_q = (int32_t*)take(kWMaxQ * 4);
    a.ws.f_c = (int32_t*)take(kWMaxQ * 4);
    a.ws.g_src = (int32_t*)take(kWMaxQ * 4);
    a.ws.g_end = (int32_t*)take(kWMaxQ * 4);
    a.ws.g_len = (int32_t*)take(kWMaxQ * 4);
    a.ws.g_last = (int32_t*)take(kWMaxQ * 4);
    a.ws.g_tail = (uint32_t*)take(kWMaxQ * 16);
    a.ws.g_lbl = (uint32_t*)take(kWMaxQ * 32);
    a.ws.ssum = (uint32_t*)take(nm * 8);
    a.ws.org = (int32_t*)take((size_t)emax * 4);
    a.ws.esum = (uint32_t*)take((size_t)emax * 8);
    a.ws.bits = (uint32_t*)take((size_t)emax * W * 4);
    a.rec.col_gap = (uint8_t*)take(nm);
    a.rec.e_dst = (int32_t*)take((size_t)edge_cap * 4);
    a.rec.e_src = (int32_t*)take((size_t)edge_cap * 4);
    a.rec.e_lbl = (uint32_t*)take((size_t)edge_cap * 32);
    a.rec.gap_col = (int32_t*)take((size_t)n * 4);
    a.rec.pre_col = (int32_t*)take((size_t)n * 4);
    a.rec.post_col = (int32_t*)take((size_t)n * 4);
    a.rec.cnt = (uint32_t*)take((size_t)emax * VW * 4);
    a.rec.meta = (int32_t*)take(32);
    a.rec.edge_cap = edge_cap;
    a.rec.n_edges = 0;
    a.good = (uint32_t*)take((size_t)emax * W * 4);
    a.last_col = (int32_t*)take(nm * 4);
    a.in_off = (int32_t*)take((nm + 1) * 4);
    a.out_off = (int32_t*)take((nm + 1) * 4);
    a.succ_off = (int32_t*)take((nm + 1) * 4);
    a.out_idx = (int32_t*)take((size_t)edge_cap * 4);
    a.succ_idx = (int32_t*)take((size_t)emax * 4);
    a.expn = (uint32_t*)take(nm * W * 4);
    a.eidx = (int32_t*)take(nm * (nm + 1) / 2 * 4);
    a.gnz = (uint8_t*)take((size_t)emax);
    a.cursor = (int32_t*)take(2 * (nm + 1) * 4);
    a.key_q = (int32_t*)take(kMaxQ * 4);
    a.bexpn = (uint32_t*)take(nm * W * 4);
    a.bnew = (uint32_t*)take(nm * VW * 4);
    return a;
  }
};

// meta slots of a sequence's record
enum { M_NCOLS = 0, M_NEDGES = 1, M_START = 2, M_ACCEPT = 3, M_STATUS = 4, M_NENT = 5 };

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

// The same forward charts with a whole CTA per sequence: the block walk
// spreads each closure round's dirty origins and completion pairs over the
// warps (for long sequences of wide grammars, where one warp's walk is a long
// serial chain).  Selected with EPIC_FORWARD_BLOCK=1.
__global__ void __launch_bounds__(kThreads) k_forward_block(DevGrammar g, const LexEntry* __restrict__ table,
                                                            int vocab, const int32_t* __restrict__ x, int B, int n,
                                                            SeqPack sp, unsigned long long* stats) {
  __shared__ WalkShared sh;
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
    sc.expn = a.bexpn;
    sc.bnew = a.bnew;
    const BlockRec br{a.rec.col_gap, a.rec.e_dst,   a.rec.e_src,   a.rec.e_lbl,    a.rec.cnt,
                      a.ws.esum,     a.rec.gap_col, a.rec.pre_col, a.rec.post_col, a.rec.edge_cap};
    WsDims d;
    d.nmax = sp.nmax;
    d.emax = sp.emax;
    EarleyColsT<true> cols(g, table, ws, sc, d, sh);
    cols.rec = &br;
    Walk<EarleyColsT<true>> walk(cols, g, table, sc, sh, vocab);
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

// ------------------------------------------------------------------ 2. good masks
// warp: dst |= src >> 1 over W words ((item i+1 good) => candidate i)
__device__ __forceinline__ uint32_t shr1_word(const uint32_t* src, int w, int W) {
  uint32_t v = src[w] >> 1;
  if (w + 1 < W) v |= src[w + 1] << 31;
  return v;
}

constexpr int kGoodWarps = 32;  // one CTA per sequence

// Good items of a sequence's forward chart, columns from last to first.
// Item i of entry (j, o) is good when it is present and
//  - it is the accepting item at the accept node with the start origin;
//  - an out-edge j -> j2 scans a terminal it expects (or is epsilon) and the
//    advanced item of (j2, o) is good;
//  - it waits on a nonterminal that completes from origin j at column j2
//    (j2 = j: a nullable one) and the advanced item of (j2, o) is good;
//  - j is a gap and the item advanced over any symbol is good;
//  - it is complete with left side B, and some item of column o, origin o2,
//    waiting on B has its advanced item good at (j, o2).
// The first three read later columns only (final); the last two read this
// column: its entries iterate to the least fixpoint together.
__global__ void __launch_bounds__(32 * kGoodWarps, 1) k_good(DevGrammar g, int B, SeqPack sp) {
  const long long b = blockIdx.x;
  if (b >= B) return;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nthr = blockDim.x;
  const int W = g.W, VW = g.VW;
  SeqArena a = sp.carve(b);
  int32_t* meta = a.rec.meta;
  if (meta[M_STATUS] != 1) return;
  const int N = meta[M_NCOLS], NE = meta[M_NEDGES];
  const int32_t* col = a.ws.col_off;
  const int32_t* org = a.ws.org;
  const int start = meta[M_START], accept = meta[M_ACCEPT];
  __shared__ int s_flag, s_self;
  __shared__ uint32_t s_nt[kGoodWarps][kWMaxVW];
  constexpr int KW = kWMaxW / 32;  // item words per lane
  int32_t* cur_o = a.cursor;          // [N + 1]
  int32_t* cur_s = a.cursor + N + 1;  // [N + 1]
  // edges by source and entries by origin (CSR), entry index by (column, origin)
  for (int j = tid; j <= N; j += nthr) {
    a.in_off[j] = 0;
    a.out_off[j] = 0;
    a.succ_off[j] = 0;
  }
  for (int u = tid; u < N; u += nthr) a.last_col[u] = -1;
  const size_t ntri = (size_t)N * (N + 1) / 2;
  for (size_t q = tid; q < ntri; q += nthr) a.eidx[q] = -1;
  __syncthreads();
  for (int e = tid; e < NE; e += nthr) {
    atomicAdd(&a.in_off[a.rec.e_dst[e] + 1], 1);
    atomicAdd(&a.out_off[a.rec.e_src[e] + 1], 1);
  }
  for (int j = warp; j < N; j += kGoodWarps)
    for (long long k = col[j] + lane; k < col[j + 1]; k += 32) {
      const int o = org[k];
      a.eidx[tri_index(j, o)] = (int32_t)k;
      a.gnz[k] = 0;
      atomicAdd(&a.succ_off[o + 1], 1);
      atomicMax(&a.last_col[o], j);
    }
  __syncthreads();
  if (tid == 0)
    for (int j = 0; j < N; ++j) {
      a.in_off[j + 1] += a.in_off[j];
      a.out_off[j + 1] += a.out_off[j];
      a.succ_off[j + 1] += a.succ_off[j];
    }
  __syncthreads();
  for (int j = tid; j < N; j += nthr) {
    cur_o[j] = a.out_off[j];
    cur_s[j] = a.succ_off[j];
  }
  __syncthreads();
  for (int e = tid; e < NE; e += nthr) a.out_idx[atomicAdd(&cur_o[a.rec.e_src[e]], 1)] = e;
  for (int j = warp; j < N; j += kGoodWarps)
    for (long long k = col[j] + lane; k < col[j + 1]; k += 32) a.succ_idx[atomicAdd(&cur_s[org[k]], 1)] = j;
  __syncthreads();

  uint32_t* G = a.good;
  uint32_t* sfold = (uint32_t*)a.cursor;  // per successor of the column (the cursors are free now)
  const int nwl = (W + 31) >> 5;          // item words per lane in use
  for (int j = N - 1; j >= 0; --j) {
    const int s0 = a.succ_off[j], s1 = a.succ_off[j + 1];
    const bool gap = a.rec.col_gap[j] != 0;
    const long long k0 = col[j], k1 = col[j + 1];
    if (k0 == k1) continue;
    // EXPN of what completes from origin j at each column j2 (j2 = j included)
    if (tid == 0) s_self = -1;
    __syncthreads();
    for (int si = s0 + tid; si < s1; si += nthr)
      if (a.succ_idx[si] == j) s_self = si - s0;
    __syncthreads();
    const int self_si = s_self;
    for (int si = s0 + warp; si < s1; si += kGoodWarps) {
      const int j2 = a.succ_idx[si];
      const uint32_t* cn = a.rec.cnt + (size_t)a.eidx[tri_index(j2, j)] * VW;
      expn_of_set(g, cn, a.expn + (size_t)(si - s0) * W);
      if (lane == 0) {  // folded set (bit C mod 32): a filter against an entry's waited nonterminals
        uint32_t f = 0;
        for (int v = 0; v < VW; ++v) f |= cn[v];
        sfold[si - s0] = f;
      }
    }
    __syncthreads();
    // from the later columns: scans along the out-edges, nested constituents
    // (the lanes look up 32 successor columns at a time)
    for (long long k = k0 + warp; k < k1; k += kGoodWarps) {
      const int o = org[k];
      const uint32_t* bits = a.ws.bits + (size_t)k * W;
      uint32_t* Gk = G + (size_t)k * W;
      uint32_t acc[KW];
#pragma unroll
      for (int i = 0; i < KW; ++i) acc[i] = 0;
      if (j == accept && o == start && lane == ((g.accept_item >> 5) & 31))
        acc[g.accept_item >> 10] |= 1u << (g.accept_item & 31);
      for (int ei = a.out_off[j]; ei < a.out_off[j + 1]; ++ei) {
        const int e = a.out_idx[ei];
        const int k2 = a.eidx[tri_index(a.rec.e_dst[e], o)];
        if (k2 < 0 || !a.gnz[k2]) continue;
        const uint32_t* G2 = G + (size_t)k2 * W;
        const uint32_t* L = a.rec.e_lbl + (size_t)e * 8;
        uint32_t lw8[8];
        bool eps = true;
        for (int lw = 0; lw < 8; ++lw) {
          lw8[lw] = L[lw];
          eps &= lw8[lw] == 0;
        }
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          if (i >= nwl) break;
          const int w = lane + 32 * i;
          if (w < W) {
            if (eps) {
              acc[i] |= G2[w];
            } else {
              uint32_t m = 0;
              for (int lw = 0; lw < 8; ++lw) {
                uint32_t lm = lw8[lw];
                while (lm) {
                  const int bb = __ffs(lm) - 1;
                  lm &= lm - 1;
                  const int t = (lw << 5) + bb;
                  if (t < g.T) m |= g.exp_term[(size_t)t * W + w];
                }
              }
              acc[i] |= m & shr1_word(G2, w, W);
            }
          }
        }
      }
      const uint32_t wfold = a.ws.esum[(size_t)k * 2];  // waited nonterminals, folded
      for (int sb = s0; sb < s1; sb += 32) {
        const int si = sb + lane;
        int k3 = -1;
        if (si < s1 && si - s0 != self_si && (sfold[si - s0] & wfold) != 0) {
          const int kk = a.eidx[tri_index(a.succ_idx[si], o)];
          if (kk >= 0 && a.gnz[kk]) k3 = kk;
        }
        unsigned act = __ballot_sync(0xffffffffu, k3 >= 0);
        while (act) {
          const int l = __ffs(act) - 1;
          act &= act - 1;
          const int kk = __shfl_sync(0xffffffffu, k3, l);
          const uint32_t* ex = a.expn + (size_t)(sb + l - s0) * W;
          const uint32_t* G3 = G + (size_t)kk * W;
#pragma unroll
          for (int i = 0; i < KW; ++i) {
            if (i >= nwl) break;
            const int w = lane + 32 * i;
            if (w < W) acc[i] |= ex[w] & shr1_word(G3, w, W);
          }
        }
      }
      bool nz = false;
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        if (w < W) {
          const uint32_t v = bits[w] & acc[i];
          Gk[w] = v;
          nz |= v != 0;
        }
      }
      nz = __any_sync(0xffffffffu, nz);
      if (lane == 0) a.gnz[k] = nz ? 1 : 0;
    }
    __syncthreads();
    // completions within the column and the self rules, to the fixpoint
    for (int pass = 0;; ++pass) {
      if (pass > (1 << 20)) {  // cannot happen before the fixpoint; never silently wrong
        if (tid == 0) meta[M_STATUS] = -1;
        return;
      }
      if (tid == 0) s_flag = 0;
      __syncthreads();
      bool changed = false;
      uint32_t* bset = s_nt[warp];
      for (long long k = k0 + warp; k < k1; k += kGoodWarps) {
        const int o = org[k];
        const uint32_t* bits = a.ws.bits + (size_t)k * W;
        uint32_t* Gk = G + (size_t)k * W;
        // each round that changes the entry adds an item
        for (int round = 0; round <= W * 32; ++round) {
          for (int v = lane; v < VW; v += 32) bset[v] = 0;
          __syncwarp();
          for (long long kb = col[o]; kb < col[o + 1]; kb += 32) {  // 32 lookups at a time
            const long long kp = kb + lane;
            long long kk = -1;
            if (kp < col[o + 1]) {
              const int o2 = org[kp];
              kk = (o2 == o) ? k : a.eidx[tri_index(j, o2)];
              if (kk >= 0 && kk != k && !a.gnz[kk]) kk = -1;
            }
            unsigned act = __ballot_sync(0xffffffffu, kk >= 0);
            while (act) {
              const int l = __ffs(act) - 1;
              act &= act - 1;
              const long long kq = __shfl_sync(0xffffffffu, kk, l);
              const uint32_t* P = a.ws.bits + (size_t)(kb + l) * W;
              const uint32_t* GK = G + (size_t)kq * W;
              for (int w = lane; w < W; w += 32) {
                uint32_t m = P[w] & g.any_nt[w] & shr1_word(GK, w, W);
                while (m) {
                  const int bb = __ffs(m) - 1;
                  m &= m - 1;
                  const int Bn = g.item_next[(w << 5) + bb] - g.T;
                  atomicOr(&bset[Bn >> 5], 1u << (Bn & 31));
                }
              }
            }
          }
          __syncwarp();
          bool ch = false;
          for (int w = lane; w < W; w += 32) {
            uint32_t add = 0;
            uint32_t m = bits[w] & g.complete[w];
            while (m) {
              const int bb = __ffs(m) - 1;
              m &= m - 1;
              const int L2 = g.item_lhs[(w << 5) + bb];
              if ((bset[L2 >> 5] >> (L2 & 31)) & 1u) add |= 1u << bb;
            }
            const uint32_t s = shr1_word(Gk, w, W);
            if (gap) add |= g.next_any[w] & s;
            if (self_si >= 0) add |= a.expn[(size_t)self_si * W + w] & s;
            add &= bits[w];
            const uint32_t old = Gk[w];
            if ((old | add) != old) {
              Gk[w] = old | add;
              ch = true;
            }
          }
          if (!__any_sync(0xffffffffu, ch)) break;
          changed = true;
          if (lane == 0) a.gnz[k] = 1;
        }
      }
      if (changed && lane == 0) s_flag = 1;
      __syncthreads();
      const int more = s_flag;
      __syncthreads();
      if (!more) break;
    }
  }
}

// ------------------------------------------------------------------ 3. checks by region
template <bool SM>
struct RegionCheck {
  WarpWalker<SM, true>& w;
  SeqArena& a;
  int32_t* fmap;     // [nmax] F node -> own column with carried rows (-1)
  int32_t* act;      // [nmax] own columns whose rows wait on nonterminals
  int32_t* act_f;    // [nmax] their F node

  // x (+) {(i, t)}: 1 valid, 0 invalid, -1 capacity
  __device__ int run(const int32_t* x, int n, int i, int t) {
    const int lane = threadIdx.x & 31;
    const int32_t* meta = a.rec.meta;
    const int NF = meta[M_NCOLS];
    // base chart
    w.base_cols = NF;
    w.base_ent = a.ws.col_off[NF];
    w.b_col_off = a.ws.col_off;
    w.b_org = a.ws.org;
    w.b_bits = a.ws.bits;
    w.b_esum = a.ws.esum;
    w.good = a.good;
    w.b_eidx = a.eidx;
    w.accept_node = meta[M_ACCEPT];
    w.ncols = NF;
    w.nent = 0;
    w.status = 0;
    w.nf = 0;
    w.found = 0;
    w.suffix_mode = false;
    w.region_start = -1;
    if (lane == 0) w.ws.col_off[0] = 0;
    __syncwarp();
    // the mask run [ra, rb] holding i
    int ra = i, rb = i;
    while (ra > 0 && x[ra - 1] < 0) --ra;
    while (rb + 1 < n && x[rb + 1] < 0) ++rb;
    int start = meta[M_START];
    int src;
    bool at_begin;
    int left_lo = 0, left_hi = 0;  // fixed tokens before t in the span
    if (i > ra) {
      src = a.rec.gap_col[i];  // the left part of the run is the whole run's gap
      at_begin = false;
    } else if (ra > 0) {
      int s = ra - 1;
      while (s > 0 && x[s - 1] >= 0) --s;
      src = a.rec.pre_col[ra - 1];
      at_begin = s == 0;
      left_lo = s;
      left_hi = ra;
    } else {  // t starts the output: a BEGIN node of the check's own
      int c = w.open_column();
      if (c < 0) return -1;
      w.seed(c);
      w.close_column(c, false);
      w.finish_column(c);
      if (w.status) return -1;
      src = c;
      at_begin = true;
      start = c;
      w.region_start = c;
    }
    int right_lo = 0, right_hi = 0;
    bool to_end;
    int rf;  // F node after the region
    if (i < rb) {
      to_end = false;
      rf = a.rec.gap_col[i];
    } else if (rb + 1 < n) {
      int e = rb + 1;
      while (e + 1 < n && x[e + 1] >= 0) ++e;
      right_lo = rb + 1;
      right_hi = e + 1;
      to_end = (e == n - 1);
      rf = to_end ? -1 : a.rec.post_col[rb + 1];
    } else {
      to_end = true;
      rf = -1;
    }
    w.start_col = start;
    w.frontier_from(src, at_begin);
    for (int p = left_lo; p < left_hi && w.nf > 0; ++p)
      if (!w.span_step(x[p])) return -1;
    if (w.nf > 0 && !w.span_step(t)) return -1;
    for (int p = right_lo; p < right_hi && w.nf > 0; ++p)
      if (!w.span_step(x[p])) return -1;
    if (w.nf == 0) return 0;
    if (to_end) {
      int c = w.end_from_frontier();
      if (c < 0) return -1;
      w.close_column(c, false);
      w.finish_column(c);
      if (w.status) return -1;
      return w.accepts(c, start) ? 1 : 0;
    }
    // the node after the region, then the suffix, carrying only the items
    // whose origin is a node of the region
    for (int j = lane; j < NF; j += 32) fmap[j] = -1;
    __syncwarp();
    int nact = 0;
    w.suffix_mode = true;
    w.res_node = rf;
    {
      int c = w.gap_from_frontier();
      if (c < 0) return -1;
      w.close_column(c, true);
      w.finish_column(c);
      if (w.status) return -1;
      if (w.found) return 1;
      if (!w.column_empty(c)) {
        if (lane == 0) {
          fmap[rf] = c;
          act[0] = c;
          act_f[0] = rf;
        }
        __syncwarp();
        nact = 1;
      }
    }
    if (nact == 0) return 0;  // nothing of the region passes the node after it (a gap)
    for (int j = rf + 1; j < NF; ++j) {
      int c = w.open_column();
      if (c < 0) return -1;
      w.res_node = j;
      // arrivals along F's edges into j from nodes that carry rows
      for (int e = a.in_off[j]; e < a.in_off[j + 1]; ++e) {
        int oc = fmap[a.rec.e_src[e]];
        if (oc < 0) continue;
        const uint32_t* L = a.rec.e_lbl + (size_t)e * 8;
        bool eps = true;
        for (int lw = 0; lw < 8; ++lw) eps &= L[lw] == 0;
        if (eps) {
          w.arrive(oc, nullptr, false);
        } else {
          w.label_set(L);
          w.arrive(oc, w.sh.lbl, true);
        }
      }
      // nested constituents from an earlier carrying node u completing at j
      for (int ai = 0; ai < nact; ++ai) {
        int u = act[ai], uf = act_f[ai];
        long long kc = w.find_base(j, uf);
        if (kc < 0) continue;
        for (int v = lane; v < w.VW; v += 32) w.sh.nt[v] = a.rec.cnt[(size_t)kc * w.VW + v];
        __syncwarp();
        uint32_t fold = 0;
        for (int v = 0; v < w.VW; ++v) fold |= w.sh.nt[v];
        if (!fold) continue;
        expn_of_set(w.g, w.sh.nt, w.sh.expn);
        __syncwarp();
        w.scatter(u, w.sh.expn, true, 0, fold);
        if (w.status) return -1;
      }
      w.close_column(c, a.rec.col_gap[j] != 0);
      w.finish_column(c);
      if (w.status) return -1;
      if (w.found) return 1;
      bool keep = !w.column_empty(c);
      if (keep && lane == 0) fmap[j] = c;
      // carrying nodes whose F origin can no longer complete anything retire
      int na = 0;
      for (int ai = 0; ai < nact; ++ai) {
        int uf = act_f[ai];
        if (a.last_col[uf] > j) {
          if (lane == 0) {
            act[na] = act[ai];
            act_f[na] = uf;
          }
          ++na;
        }
      }
      if (keep && a.last_col[j] > j) {
        if (lane == 0) {
          act[na] = c;
          act_f[na] = j;
        }
        ++na;
      }
      __syncwarp();
      nact = na;
      // a gap is a cut of the graph: if nothing is carried through it and no
      // earlier node can still complete past it, nothing of the region comes back
      if (!keep && a.rec.col_gap[j] && nact == 0) break;
    }
    return w.found ? 1 : 0;
  }
};

// per-warp tables of a region check
struct RegScratch {
  int32_t* fmap;
  int32_t* act;
  int32_t* act_f;
};

template <bool SM>
__global__ void __launch_bounds__(32 * kWarpsPerCta) k_check(
    DevGrammar g, const LexEntry* __restrict__ table, int vocab, const int32_t* __restrict__ x, int n,
    const int32_t* __restrict__ pos, int k, const int32_t* __restrict__ cand, int K, long long total,
    uint8_t* __restrict__ valid, SeqPack sp, WPack wp, int32_t* __restrict__ regs, int rmax,
    unsigned long long* counter, unsigned long long* stats) {
  __shared__ WSh shm[kWarpsPerCta];
  extern __shared__ __align__(16) unsigned char dyn[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  WSh& sh = shm[warp];
  for (int w = lane; w < kWCols / 32; w += 32) {
    sh.touched[w] = 0;
    sh.dirty[w] = 0;
  }
  for (int v = lane; v < kWMaxVW; v += 32) {
    sh.vset[v] = 0;
    sh.vdone[v] = 0;
  }
  __syncwarp();
  const long long gw = (long long)blockIdx.x * (blockDim.x >> 5) + warp;
  WarpWalker<SM, true> walk(g, table, wp.carve(gw), sh, wp.nmax, wp.emax, vocab);
  if constexpr (SM) {
    size_t per = smem_per_warp(wp.nmax, rmax, g.W, g.VW);
    unsigned char* base = dyn + per * warp;
    uint32_t* rows = (uint32_t*)base;
    uint32_t* bd = rows + (size_t)rmax * g.W;
    int32_t* sorg = (int32_t*)(bd + (size_t)rmax * g.VW);
    uint32_t* ssum = (uint32_t*)(sorg + rmax);
    int16_t* so = (int16_t*)(ssum + 2 * rmax);
    walk.set_smem(rows, bd, so, sorg, ssum, rmax);
  }
  RegScratch rs;
  rs.fmap = regs + (size_t)gw * 3 * wp.nmax;
  rs.act = rs.fmap + wp.nmax;
  rs.act_f = rs.act + wp.nmax;
  unsigned long long n_checks = 0, n_valid = 0, n_ovf = 0, n_bad = 0, n_cols = 0, n_ent = 0;
  for (;;) {
    long long jb = 0;
    if (lane == 0) jb = (long long)atomicAdd(counter, 1ull);
    jb = __shfl_sync(0xffffffffu, jb, 0);
    if (jb >= total) break;
    long long b = jb / ((long long)k * K);
    long long jj = (jb / K) % k;
    const int32_t* xb = x + b * n;
    int i = pos[b * k + jj], t = cand[jb];
    int r;
    long long own_cols = 0, own_ent = 0;  // columns and entries this check stored
    if (i < 0 || i >= n || xb[i] >= 0 || t < 0 || t >= vocab) {
      r = -2;
    } else {
      SeqArena a = sp.carve(b);
      int fs = a.rec.meta[M_STATUS];
      if (fs == 0) {
        r = 0;  // x is not completable, so no update of it is
      } else if (fs == 1) {
        RegionCheck<SM> rc{walk, a, rs.fmap, rs.act, rs.act_f};
        r = rc.run(xb, n, i, t);
        if (r < 0) walk.cleanup();
        own_cols = walk.ncols - walk.base_cols;
        own_ent = walk.nent;
      } else {  // the sequence's forward chart did not fit: walk the whole check
        walk.base_cols = 0;
        walk.base_ent = 0;
        walk.suffix_mode = false;
        r = walk.run(xb, n, i, t);
        own_cols = walk.ncols;
        own_ent = walk.nent;
      }
      walk.base_cols = 0;
      walk.base_ent = 0;
      walk.suffix_mode = false;
    }
    if (lane == 0) valid[jb] = r == 1 ? 1 : (r == -1 ? 2 : 0);
    ++n_checks;
    n_valid += r == 1;
    n_ovf += r == -1;
    n_bad += r == -2;
    n_cols += own_cols;
    n_ent += own_ent;
  }
  if (lane == 0 && n_checks) {
    atomicAdd(&stats[0], n_checks);
    atomicAdd(&stats[1], n_valid);
    atomicAdd(&stats[2], n_ovf);
    atomicAdd(&stats[3], n_bad);
    atomicAdd(&stats[4], n_cols);
    atomicAdd(&stats[5], n_ent);
  }
}

}  // namespace epic

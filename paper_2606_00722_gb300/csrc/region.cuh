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
           r((size_t)emax * 4) + r(nm * W * 4);
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
    return a;
  }
};

// meta slots of a sequence's record
enum { M_NCOLS = 0, M_NEDGES = 1, M_START = 2, M_ACCEPT = 3, M_STATUS = 4, M_NENT = 5 };

// ------------------------------------------------------------------ 1. forward chart
template <bool SM>
__global__ void __launch_bounds__(32 * kWarpsPerCta) k_forward(DevGrammar g, const LexEntry* __restrict__ table,
                                                                int vocab, const int32_t* __restrict__ x, int B, int n,
                                                                SeqPack sp, int rmax) {
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
  WarpWalker<SM> walk(g, table, a.ws, sh, sp.nmax, sp.emax, vocab);
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
  }
}

// ------------------------------------------------------------------ 2. good masks
// warp: dst |= src >> 1 over W words ((item i+1 good) => candidate i)
__device__ __forceinline__ uint32_t shr1_word(const uint32_t* src, int w, int W) {
  uint32_t v = src[w] >> 1;
  if (w + 1 < W) v |= src[w + 1] << 31;
  return v;
}

__global__ void __launch_bounds__(32 * kWarpsPerCta) k_good(DevGrammar g, int B, SeqPack sp) {
  int warp = threadIdx.x >> 5;
  long long b = (long long)blockIdx.x * (blockDim.x >> 5) + warp;
  if (b >= B) return;
  const int lane = threadIdx.x & 31;
  const int W = g.W, VW = g.VW;
  SeqArena a = sp.carve(b);
  const int32_t* meta = a.rec.meta;
  if (meta[M_STATUS] != 1) return;
  const int N = meta[M_NCOLS], NE = meta[M_NEDGES];
  const int32_t* col = a.ws.col_off;
  const long long E = col[N];
  const int start = meta[M_START], accept = meta[M_ACCEPT];
  // in-edge offsets (edges are stored in target order), out-edge CSR
  for (int j = lane; j <= N; j += 32) {
    a.in_off[j] = 0;
    a.out_off[j] = 0;
    a.succ_off[j] = 0;
  }
  __syncwarp();
  for (int e = lane; e < NE; e += 32) {
    atomicAdd(&a.in_off[a.rec.e_dst[e] + 1], 1);
    atomicAdd(&a.out_off[a.rec.e_src[e] + 1], 1);
  }
  for (long long k = lane; k < E; k += 32) atomicAdd(&a.succ_off[a.ws.org[k] + 1], 1);
  __syncwarp();
  if (lane == 0)
    for (int j = 0; j < N; ++j) {
      a.in_off[j + 1] += a.in_off[j];
      a.out_off[j + 1] += a.out_off[j];
      a.succ_off[j + 1] += a.succ_off[j];
    }
  __syncwarp();
  int32_t* cur = a.last_col;  // cursor, reused below as last_col
  for (int j = lane; j < N; j += 32) cur[j] = a.out_off[j];
  __syncwarp();
  for (int e = lane; e < NE; e += 32) a.out_idx[atomicAdd(&cur[a.rec.e_src[e]], 1)] = e;
  __syncwarp();
  for (int j = lane; j < N; j += 32) cur[j] = a.succ_off[j];
  __syncwarp();
  for (int c = 0; c < N; ++c)  // column by column: each list ascends
    for (long long k = col[c] + lane; k < col[c + 1]; k += 32) a.succ_idx[atomicAdd(&cur[a.ws.org[k]], 1)] = c;
  __syncwarp();
  for (int u = lane; u < N; u += 32)
    a.last_col[u] = a.succ_off[u + 1] > a.succ_off[u] ? a.succ_idx[a.succ_off[u + 1] - 1] : -1;
  __syncwarp();
  auto find = [&](int j, int o) -> long long {
    long long lo = col[j], hi = col[j + 1];
    for (long long base = lo; base < hi; base += 32) {
      long long k = base + lane;
      bool hit = k < hi && a.ws.org[k] == o;
      unsigned m = __ballot_sync(0xffffffffu, hit);
      if (m) return base + __ffs(m) - 1;
    }
    return -1;
  };
  constexpr int KW = kWMaxW / 32;
  const int nw = (W + 31) >> 5;
  __shared__ uint32_t s_nt[kWarpsPerCta][kWMaxVW];
  uint32_t* bset = s_nt[warp];
  for (int j = N - 1; j >= 0; --j) {
    const bool gap = a.rec.col_gap[j] != 0;
    // EXPN of what completes from origin j at each later column j2
    const int s0 = a.succ_off[j], s1 = a.succ_off[j + 1];
    for (int si = s0; si < s1; ++si) {
      int j2 = a.succ_idx[si];
      long long kc = find(j2, j);
      for (int w = lane; w < W; w += 32) {
        uint32_t acc = 0;
        for (int v = 0; v < VW; ++v) {
          uint32_t m = a.rec.cnt[(size_t)kc * VW + v];
          while (m) {
            int bb = __ffs(m) - 1;
            m &= m - 1;
            acc |= g.exp_nt[(size_t)((v << 5) + bb) * W + w];
          }
        }
        a.expn[(size_t)(si - s0) * W + w] = acc;
      }
    }
    __syncwarp();
    for (long long k = col[j]; k < col[j + 1]; ++k) {
      const int o = a.ws.org[k];
      const uint32_t* bits = a.ws.bits + (size_t)k * W;
      uint32_t* G = a.good + (size_t)k * W;
      for (int w = lane; w < W; w += 32) G[w] = 0;
      __syncwarp();
      if (j == accept && o == start && lane == 0)
        G[g.accept_item >> 5] = bits[g.accept_item >> 5] & (1u << (g.accept_item & 31));
      __syncwarp();
      // each round that changes the row adds an item: W * 32 + 1 rounds reach the fixpoint
      for (int round = 0; round <= W * 32; ++round) {
        bool ch = false;
        uint32_t acc[KW];
#pragma unroll
        for (int i = 0; i < KW; ++i) acc[i] = 0;
        // (ii) scans and epsilon moves along the out-edges
        for (int ei = a.out_off[j]; ei < a.out_off[j + 1]; ++ei) {
          int e = a.out_idx[ei];
          int j2 = a.rec.e_dst[e];
          long long k2 = find(j2, o);
          if (k2 < 0) continue;
          const uint32_t* G2 = a.good + (size_t)k2 * W;
          const uint32_t* L = a.rec.e_lbl + (size_t)e * 8;
          bool eps = true;
          for (int lw = 0; lw < 8; ++lw) eps &= L[lw] == 0;
#pragma unroll
          for (int i = 0; i < KW; ++i) {
            int w = lane + 32 * i;
            if (i < nw && w < W) {
              uint32_t m = 0xffffffffu;
              if (!eps) {
                m = 0;
                for (int lw = 0; lw < 8; ++lw) {
                  uint32_t lm = L[lw];
                  while (lm) {
                    int bb = __ffs(lm) - 1;
                    lm &= lm - 1;
                    int t = (lw << 5) + bb;
                    if (t < g.T) m |= g.exp_term[(size_t)t * W + w];
                  }
                }
                acc[i] |= bits[w] & m & shr1_word(G2, w, W);
              } else {
                acc[i] |= bits[w] & G2[w];
              }
            }
          }
        }
        // (iv) nested constituents completing from j at j2 (j2 = j: this row)
        for (int si = s0; si < s1; ++si) {
          int j2 = a.succ_idx[si];
          long long k3 = (j2 == j) ? k : find(j2, o);
          if (k3 < 0) continue;
          const uint32_t* G3 = a.good + (size_t)k3 * W;
#pragma unroll
          for (int i = 0; i < KW; ++i) {
            int w = lane + 32 * i;
            if (i < nw && w < W) acc[i] |= bits[w] & a.expn[(size_t)(si - s0) * W + w] & shr1_word(G3, w, W);
          }
        }
        // inside a gap every item advances over any symbol
        if (gap) {
#pragma unroll
          for (int i = 0; i < KW; ++i) {
            int w = lane + 32 * i;
            if (i < nw && w < W) acc[i] |= bits[w] & g.next_any[w] & shr1_word(G, w, W);
          }
        }
        // (v) completion: the items of column o waiting on the completed
        // nonterminal advance to good items of this node
        for (int v = lane; v < VW; v += 32) bset[v] = 0;
        __syncwarp();
        for (long long kp = col[o]; kp < col[o + 1]; ++kp) {
          int o2 = a.ws.org[kp];
          long long kk = (o2 == o) ? k : find(j, o2);
          if (kk < 0) continue;
          const uint32_t* P = a.ws.bits + (size_t)kp * W;
          const uint32_t* GK = a.good + (size_t)kk * W;
          for (int w = lane; w < W; w += 32) {
            uint32_t m = P[w] & g.any_nt[w] & shr1_word(GK, w, W);
            while (m) {
              int bb = __ffs(m) - 1;
              m &= m - 1;
              int Bn = g.item_next[(w << 5) + bb] - g.T;
              atomicOr(&bset[Bn >> 5], 1u << (Bn & 31));
            }
          }
        }
        __syncwarp();
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          int w = lane + 32 * i;
          if (i < nw && w < W) {
            uint32_t m = bits[w] & g.complete[w];
            uint32_t add = 0;
            while (m) {
              int bb = __ffs(m) - 1;
              m &= m - 1;
              int L2 = g.item_lhs[(w << 5) + bb];
              if ((bset[L2 >> 5] >> (L2 & 31)) & 1u) add |= 1u << bb;
            }
            acc[i] |= add;
          }
        }
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          int w = lane + 32 * i;
          if (i < nw && w < W) {
            uint32_t old = G[w];
            if ((old | acc[i]) != old) {
              G[w] = old | acc[i];
              ch = true;
            }
          }
        }
        __syncwarp();
        if (!__any_sync(0xffffffffu, ch)) break;
      }
    }
  }
}

// ------------------------------------------------------------------ 3. checks by region
template <bool SM>
struct RegionCheck {
  WarpWalker<SM>& w;
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
        for (int ww = lane; ww < w.W; ww += 32) {
          uint32_t acc = 0;
          for (int v = 0; v < w.VW; ++v) {
            uint32_t m = w.sh.nt[v];
            while (m) {
              int bb = __ffs(m) - 1;
              m &= m - 1;
              acc |= w.g.exp_nt[(size_t)((v << 5) + bb) * w.W + ww];
            }
          }
          w.sh.expn[ww] = acc;
        }
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
  WarpWalker<SM> walk(g, table, wp.carve(gw), sh, wp.nmax, wp.emax, vocab);
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
      } else {  // the sequence's forward chart did not fit: walk the whole check
        walk.base_cols = 0;
        walk.base_ent = 0;
        walk.suffix_mode = false;
        r = walk.run(xb, n, i, t);
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
    n_cols += walk.ncols;
    n_ent += walk.nent;
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

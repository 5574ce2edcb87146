// Checks by region, step 2: the good-item masks of each forward chart, with
// the launcher.
#include <cuda_runtime.h>

#include "launch.h"
#include "region.cuh"

namespace epic {

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


void launch_good(dim3 grid, cudaStream_t st, const DevGrammar& g, int B, const SeqPack& sp) {
  k_good<<<grid, 32 * kGoodWarps, 0, st>>>(g, B, sp);
}

int good_warps() { return kGoodWarps; }

}  // namespace epic

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

constexpr int kGoodWarps = 16;  // one CTA per sequence

// Warp, row in registers: r |= bits & M & shr1(r) until stable -- an item is
// good when it may advance within its own row and the advanced item is good.
template <int KW>
__device__ __forceinline__ void good_in_row(uint32_t (&r)[KW], const uint32_t (&bits)[KW], const uint32_t (&M)[KW],
                                            int W) {
  const int lane = threadIdx.x & 31;
  for (int it = 0; it < 64; ++it) {
    bool ch = false;
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      if (32 * i >= W) break;
      // bit b of word w takes bit b+1 (bit 0 of word w+1 for b = 31)
      uint32_t nxt = __shfl_down_sync(0xffffffffu, r[i], 1);
      const uint32_t wrap = (i + 1 < KW) ? __shfl_sync(0xffffffffu, r[i + 1], 0) : 0u;
      if (lane == 31) nxt = wrap;
      const uint32_t s = (r[i] >> 1) | (nxt << 31);
      const uint32_t add = bits[i] & M[i] & s & ~r[i];
      ch |= add != 0;
      r[i] |= add;
    }
    if (!__any_sync(0xffffffffu, ch)) break;
  }
}

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
// The first three read later columns only (final); the in-row ones (gap,
// nullable) close each row on its own.  The last one reads entries (j, o2)
// of this column with o2 <= o, so the entries holding complete items are
// closed in ascending origin order, once each: the whole CTA gathers which
// completed nonterminals of (j, o) some waiting item of column o turns good,
// then one warp closes (j, o) with its own self-loop (the entry of column o
// with origin o maps back to (j, o)).
__global__ void __launch_bounds__(32 * kGoodWarps, 1) k_good(DevGrammar g, int B, SeqPack sp) {
  extern __shared__ __align__(16) unsigned char dyn[];
  GsTables tb;
  gs_stage_tables(g, dyn, tb);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nthr = blockDim.x;
  const int W = g.W, VW = g.VW;
  constexpr int KW = kWMaxW / 32;  // item words per lane
  __shared__ int s_self;
  __shared__ uint32_t s_cn[kWMaxVW], s_bset[kWMaxVW];
  __shared__ uint32_t s_expn[kWMaxW];
  __shared__ uint32_t s_xall[kWMaxW];
  __shared__ uint32_t s_items[kWMaxW];  // good-advanceable waiting items of the gather
  __shared__ int s_flag;
  for (long long b = blockIdx.x; b < B; b += gridDim.x) {
  PH_BEGIN(t_setup);
  SeqArena a = sp.carve(b);
  int32_t* meta = a.rec.meta;
  if (meta[M_STATUS] != 1) continue;
  const int N = meta[M_NCOLS], NE = meta[M_NEDGES];
  const int32_t* col = a.ws.col_off;
  const int32_t* org = a.ws.org;
  const int start = meta[M_START], accept = meta[M_ACCEPT];
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

  PH_END(0, t_setup);
  uint32_t* G = a.good;
  uint32_t* sfold = (uint32_t*)a.cursor;  // per successor of the column (the cursors are free now)
  for (int w = tid; w < kWMaxW; w += nthr) s_items[w] = 0;
  __syncthreads();
  for (int j = N - 1; j >= 0; --j) {
    const int s0 = a.succ_off[j], s1 = a.succ_off[j + 1];
    const bool gap = a.rec.col_gap[j] != 0;
    const long long k0 = col[j], k1 = col[j + 1];
    if (k0 == k1) continue;
    // EXPN of what completes from origin j at each column j2 (j2 = j included)
    PH_BEGIN(t_succ);
    if (tid == 0) s_self = -1;
    __syncthreads();
    for (int si = s0 + tid; si < s1; si += nthr)
      if (a.succ_idx[si] == j) s_self = si - s0;
    __syncthreads();
    const int self_si = s_self;
    for (int si = s0 + warp; si < s1; si += kGoodWarps) {
      const int j2 = a.succ_idx[si];
      const uint32_t* cn = a.rec.cnt + (size_t)a.eidx[tri_index(j2, j)] * VW;
      uint32_t f = 0;
      for (int v = 0; v < VW; ++v) f |= cn[v];
      if (f) expn_of_set(g, cn, a.expn + (size_t)(si - s0) * W);
      if (lane == 0) sfold[si - s0] = f;  // folded (bit C mod 32): 0 = nothing completes
    }
    __syncthreads();
    // union of the completion masks of the successors after j
    for (int w = tid; w < W; w += nthr) {
      uint32_t u = 0;
      for (int si = s0; si < s1; ++si)
        if (si - s0 != self_si && sfold[si - s0]) u |= a.expn[(size_t)(si - s0) * W + w];
      s_xall[w] = u;
    }
    __syncthreads();
    PH_END(1, t_succ);
    // in-row rules of this column: the gap self-loop and nullable completions
    PH_BEGIN(t_a);
    uint32_t inrow[KW];
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      const int w = lane + 32 * i;
      uint32_t m = 0;
      if (w < W) {
        if (gap) m |= tb.next_any[w];
        if (self_si >= 0 && sfold[self_si]) m |= a.expn[(size_t)self_si * W + w];
      }
      inrow[i] = m;
    }
    // A. the rules that read later columns, then the in-row closure (one warp
    //    per entry)
    for (long long k = k0 + warp; k < k1; k += kGoodWarps) {
      const int o = org[k];
      const uint32_t* bp = a.ws.bits + (size_t)k * W;
      uint32_t acc[KW], bits[KW];
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        acc[i] = 0;
        bits[i] = (w < W) ? bp[w] : 0u;
      }
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
      // the most the nested rule can make good: items waiting on a
      // nonterminal that completes from j somewhere after j
      uint32_t want[KW];
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        want[i] = (w < W) ? (bits[i] & s_xall[w]) : 0u;
      }
      for (int sb = s0; sb < s1; sb += 32) {
        bool open = false;
#pragma unroll
        for (int i = 0; i < KW; ++i) open |= (want[i] & ~acc[i]) != 0;
        if (!__any_sync(0xffffffffu, open)) break;
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
            const int w = lane + 32 * i;
            if (w < W) {
              const uint32_t xw = ex[w];
              if (xw) acc[i] |= xw & shr1_word(G3, w, W);
            }
          }
        }
      }
#pragma unroll
      for (int i = 0; i < KW; ++i) acc[i] &= bits[i];
      good_in_row<KW>(acc, bits, inrow, W);
      bool nz = false;
      uint32_t* Gk = G + (size_t)k * W;
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        if (w < W) Gk[w] = acc[i];
        nz |= acc[i] != 0;
      }
      nz = __any_sync(0xffffffffu, nz);
      if (lane == 0) a.gnz[k] = nz ? 1 : 0;
    }
    __syncthreads();
    PH_END(2, t_a);
    // B. completions within the column, entries with complete items in
    //    ascending origin order
    for (long long k = k0; k < k1; ++k) {
      const int o = org[k];
      const uint32_t* cn = a.rec.cnt + (size_t)k * VW;
      for (int v = tid; v < VW; v += nthr) {
        s_cn[v] = cn[v];
        s_bset[v] = 0;
      }
      if (tid == 0) {
        uint32_t f = 0;
        for (int v = 0; v < VW; ++v) f |= cn[v];
        s_flag = f != 0;
      }
      __syncthreads();
      if (!s_flag) continue;  // no complete item here
      // items waiting on a nonterminal completed at (j, o)
      for (int w = tid; w < W; w += nthr) {
        uint32_t acc = 0, m = tb.any_nt[w];
        while (m) {
          const int bb = __ffs(m) - 1;
          m &= m - 1;
          const int Bn = tb.item_next[(w << 5) + bb] - g.T;
          if ((s_cn[Bn >> 5] >> (Bn & 31)) & 1u) acc |= 1u << bb;
        }
        s_expn[w] = acc;
      }
      __syncthreads();
      PH_BEGIN(t_g);
      // which of them some entry (o, o2 < o) of column o turns good at (j, o2):
      // each warp ORs, over its entries of column o, the waiting items whose
      // advance is good into registers (one operation per word); the items
      // become nonterminals once, at the end
      const int cb = col[o], ce = col[o + 1];
      const bool self = ce > cb && org[ce - 1] == o;
      const int nent = self ? ce - cb - 1 : ce - cb;
      {
        uint32_t ex[KW], acc[KW];
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          const int w = lane + 32 * i;
          ex[i] = (w < W) ? s_expn[w] : 0u;
          acc[i] = 0u;
        }
        for (int e = warp; e < nent; e += kGoodWarps) {
          const int kp = cb + e;
          const int kk = a.eidx[tri_index(j, org[kp])];
          if (kk < 0 || !a.gnz[kk]) continue;
          const uint32_t* P = a.ws.bits + (size_t)kp * W;
          const uint32_t* GK = G + (size_t)kk * W;
          uint32_t pv[KW], gv[KW];
#pragma unroll
          for (int i = 0; i < KW; ++i) {
            const int w = lane + 32 * i;
            pv[i] = ex[i] ? (P[w] & ex[i]) : 0u;
            gv[i] = (w < W) ? GK[w] : 0u;
          }
#pragma unroll
          for (int i = 0; i < KW; ++i) {
            if (32 * i >= W) break;
            // bit b of word w takes bit b + 1 of G (bit 0 of word w + 1 for b = 31)
            uint32_t nxt = __shfl_down_sync(0xffffffffu, gv[i], 1);
            const uint32_t wrap = (i + 1 < KW) ? __shfl_sync(0xffffffffu, gv[i + 1], 0) : 0u;
            if (lane == 31) nxt = wrap;
            acc[i] |= pv[i] & ((gv[i] >> 1) | (nxt << 31));
          }
        }
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          const int w = lane + 32 * i;
          if (w < W && acc[i]) atomicOr(&s_items[w], acc[i]);
        }
      }
      __syncthreads();
      for (int w = tid; w < W; w += nthr) {
        uint32_t m = s_items[w];
        s_items[w] = 0;  // ready for the next entry
        while (m) {
          const int bb = __ffs(m) - 1;
          m &= m - 1;
          const int Bn = tb.item_next[(w << 5) + bb] - g.T;
          const uint32_t bit = 1u << (Bn & 31);
          if (!(s_bset[Bn >> 5] & bit)) atomicOr(&s_bset[Bn >> 5], bit);
        }
      }
      __syncthreads();
      PH_END(3, t_g);
      // one warp: complete items with a good left side, the in-row closure,
      // and the self-loop through the entry of column o with origin o
      PH_BEGIN(t_w);
      if (warp == 0) {
        const uint32_t* bp = a.ws.bits + (size_t)k * W;
        const uint32_t* E = self ? a.ws.bits + (size_t)(ce - 1) * W : nullptr;
        uint32_t* Gk = G + (size_t)k * W;
        uint32_t r[KW], bits[KW];
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          const int w = lane + 32 * i;
          r[i] = (w < W) ? Gk[w] : 0u;
          bits[i] = (w < W) ? bp[w] : 0u;
        }
        bool any_change = false;
        for (int round = 0; round < 64 * kWMaxW; ++round) {
          // the self entry's waiting items whose advance is good at (j, o)
          if (self) {
#pragma unroll
            for (int i = 0; i < KW; ++i) {
              if (32 * i >= W) break;
              const int w = lane + 32 * i;
              uint32_t nxt = __shfl_down_sync(0xffffffffu, r[i], 1);
              const uint32_t wrap = (i + 1 < KW) ? __shfl_sync(0xffffffffu, r[i + 1], 0) : 0u;
              if (lane == 31) nxt = wrap;
              const uint32_t sh1 = (r[i] >> 1) | (nxt << 31);
              uint32_t m = (w < W) ? (E[w] & s_expn[w] & sh1) : 0u;
              while (m) {
                const int bb = __ffs(m) - 1;
                m &= m - 1;
                const int Bn = tb.item_next[(w << 5) + bb] - g.T;
                const uint32_t bit = 1u << (Bn & 31);
                if (!(s_bset[Bn >> 5] & bit)) atomicOr(&s_bset[Bn >> 5], bit);
              }
            }
            __syncwarp();
          }
          // complete items whose left side is turned good
          bool ch = false;
#pragma unroll
          for (int i = 0; i < KW; ++i) {
            const int w = lane + 32 * i;
            uint32_t m = (w < W) ? (bits[i] & tb.complete[w] & ~r[i]) : 0u;
            while (m) {
              const int bb = __ffs(m) - 1;
              m &= m - 1;
              const int L2 = tb.item_lhs[(w << 5) + bb];
              if ((s_bset[L2 >> 5] >> (L2 & 31)) & 1u) {
                r[i] |= 1u << bb;
                ch = true;
              }
            }
          }
          if (!__any_sync(0xffffffffu, ch)) break;
          any_change = true;
          good_in_row<KW>(r, bits, inrow, W);
          if (!self) break;
        }
        if (any_change) {
          bool nz = false;
#pragma unroll
          for (int i = 0; i < KW; ++i) {
            const int w = lane + 32 * i;
            if (w < W) Gk[w] = r[i];
            nz |= r[i] != 0;
          }
          nz = __any_sync(0xffffffffu, nz);
          if (lane == 0 && nz) a.gnz[k] = 1;
        }
      }
      __syncthreads();
      PH_END(4, t_w);
    }
  }
  __syncthreads();
  }
}


void launch_good(dim3 grid, cudaStream_t st, const DevGrammar& g, int B, const SeqPack& sp) {
  const size_t dyn = gs_tables_bytes(g.D, g.W, g.adv_steps);
  cudaFuncSetAttribute(k_good, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  k_good<<<grid, 32 * kGoodWarps, dyn, st>>>(g, B, sp);
}

int good_warps() { return kGoodWarps; }

// measurement builds: this translation unit's phase counters
int phase_read_good(unsigned long long* out16, int reset) {
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

// Witness extraction (Sec. 4.4, failure recovery): a completion of the
// partial output, read off its forward chart.  One warp per sequence walks
// the derivation of the accepting item top-down, from right to left:
//
//   goal (item i, origin o, node j) = derive the symbols before the dot of
//   item i along a path o -> j of the graph.  With X the symbol before the
//   dot, i is present at (j, o) because
//     - it arrived by an epsilon edge m -> j          -> goal (i, o, m);
//     - X is a terminal scanned on an edge m -> j     -> emit X, goal (i-1, o, m);
//     - X completed from m at j, o < m < j            -> goals (q, m, j) for a
//                                                        complete item q of X
//                                                        at (j, m), then (i-1, o, m);
//   or by a step that keeps the span (o, j):
//     - j is a gap and X was advanced inside it       -> emit X (a terminal) or
//                                                        a shortest string of X,
//                                                        goal (i-1, o, j);
//     - X is nullable (not a gap)                     -> goal (i-1, o, j);
//     - X spans all of (o, j)                         -> goals (q, o, j), (i-1, o, o).
// The first three make the span shorter and are tried first.  Steps that
// keep the span could cycle (unit productions, nullable symbols), so each
// takes a rank: the items of (j, o) explained by a shorter-span step (or
// with nothing before the dot) have rank 0, and an item gets rank t + 1
// when one of the span-keeping steps explains it from items of rank <= t
// (a least fixpoint over the pair's items, computed when a goal first needs
// it).  A span-keeping step is taken only towards lower ranks, so the search
// ends; every present item has a derivation, so every goal has a step.
// Bounded by the output capacity and a step limit.
#include <cuda_runtime.h>

#include "launch.h"
#include "region.cuh"

namespace epic {

constexpr int kWitnessGoalsPerTerm = 8;  // goal slots per output terminal

struct WGoal {
  int32_t item, o, j;
};

// per sequence: goal records, the goal stack, the item ranks of one (node,
// origin) pair, a completion mask and a nonterminal set
struct WitnessScratch {
  WGoal* goals;
  int32_t* stack;
  int16_t* rank;
  uint32_t* ex;
  uint32_t* nts;
};

__host__ __device__ inline size_t witness_bytes_per_seq(int cap, int D, int W, int VW, size_t* offs) {
  auto r16 = [](size_t b) { return (b + 15) & ~(size_t)15; };
  const size_t gcap = (size_t)cap * kWitnessGoalsPerTerm;
  size_t o = 0;
  offs[0] = o;
  o += r16(gcap * sizeof(WGoal));
  offs[1] = o;
  o += r16(gcap * 4);
  offs[2] = o;
  o += r16((size_t)D * 2);
  offs[3] = o;
  o += r16((size_t)W * 4);
  offs[4] = o;
  o += r16((size_t)VW * 4);
  return o;
}

__global__ void __launch_bounds__(32 * kWarpsPerCta) k_witness(DevGrammar g, int B, SeqPack sp, int32_t* terms,
                                                                int cap, int32_t* out_len, unsigned char* scratch,
                                                                unsigned long long* stats) {
  const int lane = threadIdx.x & 31;
  const long long b = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (b >= B) return;
  SeqArena a = sp.carve(b);
  const int32_t* meta = a.rec.meta;
  int32_t* out = terms + b * (long long)cap;
  const long long gcap = (long long)cap * kWitnessGoalsPerTerm;
  const int W = g.W, VW = g.VW, T = g.T, D = g.D;
  WitnessScratch ws;
  {
    size_t offs[5];
    const size_t per = witness_bytes_per_seq(cap, D, W, VW, offs);
    unsigned char* base = scratch + (size_t)b * per;
    ws.goals = (WGoal*)(base + offs[0]);
    ws.stack = (int32_t*)(base + offs[1]);
    ws.rank = (int16_t*)(base + offs[2]);
    ws.ex = (uint32_t*)(base + offs[3]);
    ws.nts = (uint32_t*)(base + offs[4]);
  }
  WGoal* G = ws.goals;
  int32_t* S = ws.stack;
  if (meta[M_STATUS] != 1) {  // not completable (0) or its chart did not fit (-1)
    if (lane == 0) out_len[b] = meta[M_STATUS] == 0 ? -1 : -2;
    return;
  }
  const uint32_t* bits = a.ws.bits;
  auto entry = [&](int m, int o) -> int { return (o > m || o < 0) ? -1 : a.eidx[tri_index(m, o)]; };
  auto present = [&](int item, int o, int m) -> bool {
    if (item < 0) return false;
    const int k = entry(m, o);
    return k >= 0 && ((bits[(size_t)k * W + (item >> 5)] >> (item & 31)) & 1u);
  };
  auto completes = [&](int Bn, int m, int j) -> bool {  // Bn completes from m at j
    const int k = entry(j, m);
    return k >= 0 && ((a.rec.cnt[(size_t)k * VW + (Bn >> 5)] >> (Bn & 31)) & 1u);
  };
  auto first_item = [&](int i) -> bool { return i == 0 || g.item_next[i - 1] < 0; };
  auto label_zero = [&](int e) -> bool {
    bool z = true;
    for (int w = 0; w < 8; ++w) z &= a.rec.e_lbl[(size_t)e * 8 + w] == 0u;
    return z;
  };
  // ---- ranks of the items of pair (j, o) (see above); -1: not present
  constexpr int KW = kWMaxW / 32;
  auto shift1 = [&](uint32_t (&v)[KW]) {  // item i -> i + 1 over the lane-strided words
    uint32_t carry = 0;
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      uint32_t prev = __shfl_up_sync(0xffffffffu, v[i], 1);
      if (lane == 0) prev = carry;
      carry = __shfl_sync(0xffffffffu, v[i], 31);
      v[i] = (v[i] << 1) | (prev >> 31);
    }
  };
  int rj = -1, ro = -1;  // the pair whose ranks ws.rank holds
  auto compute_ranks = [&](int j, int o) {
    const int kj = entry(j, o);
    const uint32_t* Bj = bits + (size_t)kj * W;
    uint32_t R[KW], v[KW];
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      const int w = lane + 32 * i;
      uint32_t f = 0;
      if (w < W)
        for (int bb = 0; bb < 32; ++bb) {
          const int it = (w << 5) + bb;
          if (it < D && first_item(it)) f |= 1u << bb;
        }
      R[i] = f;
    }
    // steps with a shorter span: in-edges ...
    for (int e = a.in_off[j]; e < a.in_off[j + 1]; ++e) {
      const int ks = entry(a.rec.e_src[e], o);
      if (ks < 0) continue;
      const uint32_t* Bs = bits + (size_t)ks * W;
      if (label_zero(e)) {
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          const int w = lane + 32 * i;
          if (w < W) R[i] |= Bs[w];
        }
      } else {
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          const int w = lane + 32 * i;
          uint32_t m = 0;
          if (w < W)
            for (int lw = 0; lw < 8; ++lw) {
              uint32_t lm = a.rec.e_lbl[(size_t)e * 8 + lw];
              while (lm) {
                const int bb = __ffs(lm) - 1;
                lm &= lm - 1;
                const int t = (lw << 5) + bb;
                if (t < T) m |= g.exp_term[(size_t)t * W + w];
              }
            }
          v[i] = (w < W) ? (Bs[w] & m) : 0u;
        }
        shift1(v);
#pragma unroll
        for (int i = 0; i < KW; ++i) R[i] |= v[i];
      }
    }
    // ... and completions from m, o < m < j
    for (int m = o + 1; m < j; ++m) {
      const int kl = entry(m, o), kc = entry(j, m);
      if (kl < 0 || kc < 0) continue;
      const uint32_t* cn = a.rec.cnt + (size_t)kc * VW;
      uint32_t any = 0;
      for (int vv = 0; vv < VW; ++vv) any |= cn[vv];
      if (!any) continue;
      expn_of_set(g, cn, ws.ex);
      __syncwarp();
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        v[i] = (w < W) ? (bits[(size_t)kl * W + w] & ws.ex[w]) : 0u;
      }
      __syncwarp();
      shift1(v);
#pragma unroll
      for (int i = 0; i < KW; ++i) R[i] |= v[i];
    }
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      const int w = lane + 32 * i;
      R[i] = (w < W) ? (R[i] & Bj[w]) : 0u;
    }
    auto write_ranks = [&](const uint32_t (&M)[KW], int r, bool all) {
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        if (w >= W) continue;
        for (int bb = 0; bb < 32; ++bb) {
          const int it = (w << 5) + bb;
          if (it >= D) break;
          if ((M[i] >> bb) & 1u) ws.rank[it] = (int16_t)r;
          else if (all) ws.rank[it] = -1;
        }
      }
    };
    write_ranks(R, 0, true);
    // steps that keep the span, from lower ranks
    const bool gap = a.rec.col_gap[j] != 0;
    const uint32_t* ADV = gap ? g.next_any : g.nullable_next;
    const int kp = entry(o, o);
    for (int t = 1; t < 0x7fff; ++t) {
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        v[i] = (w < W) ? (R[i] & ADV[w]) : 0u;
      }
      shift1(v);
      uint32_t nw[KW];
#pragma unroll
      for (int i = 0; i < KW; ++i) nw[i] = v[i];
      // X spanning (o, j): the left sides of R's complete items
      for (int vv = lane; vv < VW; vv += 32) ws.nts[vv] = 0;
      __syncwarp();
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        uint32_t m = (w < W) ? (R[i] & g.complete[w]) : 0u;
        while (m) {
          const int bb = __ffs(m) - 1;
          m &= m - 1;
          const int L = g.item_lhs[(w << 5) + bb];
          atomicOr(&ws.nts[L >> 5], 1u << (L & 31));
        }
      }
      __syncwarp();
      expn_of_set(g, ws.nts, ws.ex);
      __syncwarp();
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        const uint32_t P = (j == o) ? R[i] : ((w < W && kp >= 0) ? bits[(size_t)kp * W + w] : 0u);
        v[i] = (w < W) ? (P & ws.ex[w]) : 0u;
      }
      __syncwarp();
      shift1(v);
      bool grew = false;
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        nw[i] = (w < W) ? ((nw[i] | v[i]) & Bj[w] & ~R[i]) : 0u;
        grew |= nw[i] != 0;
        R[i] |= nw[i];
      }
      if (!__any_sync(0xffffffffu, grew)) break;
      write_ranks(nw, t, false);
    }
    __syncwarp();
    rj = j;
    ro = o;
  };
  const int start = meta[M_START], accept = meta[M_ACCEPT];
  int len = 0, ng = 0, ns = 0, status = 0;  // status: 0 ok, 2 capacity, 3 no step found
  if (!present(g.accept_item, start, accept)) status = 3;
  if (lane == 0 && status == 0) {
    G[0] = WGoal{g.accept_item, start, accept};
    S[0] = 0;
  }
  ng = ns = status == 0 ? 1 : 0;
  __syncwarp();
  auto emit = [&](int t, bool in_gap) {
    if (len >= cap) {
      status = 2;
      return;
    }
    if (lane == 0) out[len] = t | (in_gap ? (1 << 16) : 0);
    ++len;
  };
  auto push = [&](int item, int o, int j) {
    if (ng >= gcap || ns >= gcap) {
      status = 2;
      return;
    }
    if (lane == 0) {
      G[ng] = WGoal{item, o, j};
      S[ns] = ng;
    }
    __syncwarp();
    ++ng;
    ++ns;
  };
  // a complete item of nonterminal Bn at (j, m) (rank below rmax when the
  // ranks of (j, m) are loaded), -1 if none
  auto complete_item = [&](int Bn, int m, int j, int rmax) -> int {
    const int c0 = g.nt_comp_off[Bn], c1 = g.nt_comp_off[Bn + 1];
    for (int cb = c0; cb < c1; cb += 32) {
      const int c = cb + lane;
      bool ok = c < c1 && present(g.nt_comp[c], m, j);
      if (ok && rmax >= 0) {
        const int r = ws.rank[g.nt_comp[c]];
        ok = r >= 0 && r < rmax;
      }
      const unsigned qm = __ballot_sync(0xffffffffu, ok);
      if (qm) return __shfl_sync(0xffffffffu, c < c1 ? g.nt_comp[c] : -1, __ffs(qm) - 1);
    }
    return -1;
  };
  for (long long step = 0; ns > 0 && status == 0; ++step) {
    if (step > 64ll * gcap) {
      status = 3;
      break;
    }
    const int gi = S[--ns];
    const WGoal cur = G[gi];
    const int i = cur.item, o = cur.o, j = cur.j;
    if (first_item(i)) continue;  // nothing before the dot: o reaches j by epsilon edges
    // 1. arrived by an epsilon edge
    int eps_src = -1;
    for (int eb = a.in_off[j]; eb < a.in_off[j + 1] && eps_src < 0; eb += 32) {
      const int e = eb + lane;
      const bool ok = e < a.in_off[j + 1] && label_zero(e) && present(i, o, a.rec.e_src[e]);
      const unsigned m = __ballot_sync(0xffffffffu, ok);
      if (m) eps_src = __shfl_sync(0xffffffffu, e < a.in_off[j + 1] ? a.rec.e_src[e] : -1, __ffs(m) - 1);
    }
    if (eps_src >= 0) {
      push(i, o, eps_src);
      continue;
    }
    const int X = g.item_next[i - 1];
    const bool gap = a.rec.col_gap[j] != 0;
    if (X < T) {
      // 2. scanned on a labelled edge
      int src = -1;
      for (int eb = a.in_off[j]; eb < a.in_off[j + 1] && src < 0; eb += 32) {
        const int e = eb + lane;
        bool ok = false;
        if (e < a.in_off[j + 1])
          ok = ((a.rec.e_lbl[(size_t)e * 8 + (X >> 5)] >> (X & 31)) & 1u) && present(i - 1, o, a.rec.e_src[e]);
        const unsigned m = __ballot_sync(0xffffffffu, ok);
        if (m) src = __shfl_sync(0xffffffffu, e < a.in_off[j + 1] ? a.rec.e_src[e] : -1, __ffs(m) - 1);
      }
      if (src >= 0) {
        emit(X, false);
        push(i - 1, o, src);
        continue;
      }
    } else {
      // 3. X completed from m at j, o < m < j (highest m first)
      const int Bn = X - T;
      bool found = false;
      for (int mt = j - 1; mt > o && !found; mt -= 32) {
        const int m = mt - lane;
        const bool ok = m > o && present(i - 1, o, m) && completes(Bn, m, j);
        unsigned cand = __ballot_sync(0xffffffffu, ok);
        while (cand && !found) {
          const int l = __ffs(cand) - 1;  // lowest lane = highest m
          cand &= cand - 1;
          const int mm = mt - l;
          const int q = complete_item(Bn, mm, j, -1);
          if (q >= 0) {
            push(i - 1, o, mm);  // the left part, derived after X (right to left)
            push(q, mm, j);
            found = true;
          }
        }
      }
      if (found) continue;
    }
    // 4. a step that keeps the span, towards a lower rank
    if (rj != j || ro != o) compute_ranks(j, o);
    const int r = ws.rank[i];
    if (r <= 0) {  // rank 0 has a shorter-span step, found above; -1: not present
      status = 3;
      break;
    }
    const int rp = ws.rank[i - 1];
    if (rp >= 0 && rp < r && (gap || (X >= T && ((g.nullable_next[(i - 1) >> 5] >> ((i - 1) & 31)) & 1u)))) {
      if (gap) {
        if (X < T) {
          emit(X, true);
        } else {
          for (int y = g.ny_off[X - T + 1] - 1; y >= g.ny_off[X - T] && status == 0; --y) emit(g.ny[y], true);
        }
      }
      push(i - 1, o, j);
      continue;
    }
    if (X >= T && present(i - 1, o, o) && (j != o || (rp >= 0 && rp < r))) {
      const int q = complete_item(X - T, o, j, r);
      if (q >= 0) {
        push(i - 1, o, o);
        push(q, o, j);
        continue;
      }
    }
    status = 3;
    break;
  }
  if (status == 0) {  // the terminals came right to left
    for (int t = lane; t < len / 2; t += 32) {
      const int32_t v = out[t];
      out[t] = out[len - 1 - t];
      out[len - 1 - t] = v;
    }
  }
  __syncwarp();
  if (lane == 0) {
    out_len[b] = status == 0 ? len : -2;
    if (status == 3) atomicAdd(&stats[S_WITNESS_FAIL], 1ull);
  }
}

void launch_witness(int B, cudaStream_t st, const DevGrammar& g, const SeqPack& sp, int32_t* terms, int cap,
                    int32_t* out_len, void* scratch, unsigned long long* stats) {
  const int blocks = (B + kWarpsPerCta - 1) / kWarpsPerCta;
  k_witness<<<blocks, 32 * kWarpsPerCta, 0, st>>>(g, B, sp, terms, cap, out_len, (unsigned char*)scratch, stats);
}

size_t witness_scratch_bytes(int cap, int D, int W, int VW) {
  size_t offs[5];
  return witness_bytes_per_seq(cap, D, W, VW, offs);
}

}  // namespace epic

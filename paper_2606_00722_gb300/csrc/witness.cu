// Witness extraction (Sec. 4.4, failure recovery): a completion of the
// partial output, read off its forward chart.  One warp per sequence walks
// the derivation of the accepting item top-down, from right to left:
//
//   goal (item i, origin o, node j) = derive the symbols before the dot of
//   item i along a path o -> j of the graph.  With X the symbol before the
//   dot, i is present at (j, o) because
//     - it arrived by an epsilon edge m -> j          -> goal (i, o, m);
//     - X is a terminal scanned on an edge m -> j     -> emit X, goal (i-1, o, m);
//     - j is a gap and X was advanced inside it       -> emit X (a terminal) or
//                                                        a shortest string of X,
//                                                        goal (i-1, o, j);
//     - X is nullable (not a gap)                     -> goal (i-1, o, j);
//     - X completed from m at j (m < j)               -> goals (q, m, j) for a
//                                                        complete item q of X
//                                                        at (j, m), then (i-1, o, m).
// Every item of the chart has a derivation, so each goal has one of these
// explanations; they are tried in that order, and the split m from the
// highest down, so the spans shrink.  The only step that keeps the span is
// X spanning all of [o, j]; the goal is then checked against its ancestors
// of the same span (a cycle of unit productions) and another complete item
// or split is taken.  Bounded by the output capacity and a step limit.
#include <cuda_runtime.h>

#include "launch.h"
#include "region.cuh"

namespace epic {

constexpr int kWitnessGoalsPerTerm = 8;  // goal slots per output terminal

struct WGoal {
  int32_t item, o, j, up;  // up: nearest ancestor goal with the same span (o, j), -1 if none
};

__global__ void __launch_bounds__(32 * kWarpsPerCta) k_witness(DevGrammar g, int B, SeqPack sp, int32_t* terms,
                                                                int cap, int32_t* out_len, WGoal* goals,
                                                                int32_t* stack, unsigned long long* stats) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long b = (long long)blockIdx.x * (blockDim.x >> 5) + warp;
  if (b >= B) return;
  SeqArena a = sp.carve(b);
  const int32_t* meta = a.rec.meta;
  int32_t* out = terms + b * (long long)cap;
  const long long gcap = (long long)cap * kWitnessGoalsPerTerm;
  WGoal* G = goals + b * gcap;
  int32_t* S = stack + b * gcap;
  if (meta[M_STATUS] != 1) {  // not completable (0) or its chart did not fit (-1)
    if (lane == 0) out_len[b] = meta[M_STATUS] == 0 ? -1 : -2;
    return;
  }
  const int W = g.W, VW = g.VW, T = g.T;
  const uint32_t* bits = a.ws.bits;
  auto present = [&](int item, int o, int m) -> bool {
    if (o > m || item < 0) return false;
    const int k = a.eidx[tri_index(m, o)];
    return k >= 0 && ((bits[(size_t)k * W + (item >> 5)] >> (item & 31)) & 1u);
  };
  auto completes = [&](int Bn, int m, int j) -> bool {  // Bn completes from m at j
    if (m > j) return false;
    const int k = a.eidx[tri_index(j, m)];
    return k >= 0 && ((a.rec.cnt[(size_t)k * VW + (Bn >> 5)] >> (Bn & 31)) & 1u);
  };
  auto first_item = [&](int i) -> bool { return i == 0 || g.item_next[i - 1] < 0; };
  const int start = meta[M_START], accept = meta[M_ACCEPT];
  int len = 0, ng = 0, ns = 0, status = 0;  // status: 0 ok, 2 capacity, 3 no explanation
  if (!present(g.accept_item, start, accept)) status = 3;
  if (lane == 0 && status == 0) {
    G[0] = WGoal{g.accept_item, start, accept, -1};
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
  auto push = [&](int item, int o, int j, int parent) {
    if (ng >= gcap || ns >= gcap) {
      status = 2;
      return;
    }
    // same-span ancestors are consecutive (a unit step keeps the span; any
    // other step moves an end), so the chain links only direct parents
    const int up = (parent >= 0 && G[parent].o == o && G[parent].j == j) ? parent : -1;
    if (lane == 0) {
      G[ng] = WGoal{item, o, j, up};
      S[ns] = ng;
    }
    __syncwarp();
    ++ng;
    ++ns;
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
      bool ok = false;
      if (e < a.in_off[j + 1]) {
        bool eps = true;
        for (int w = 0; w < 8; ++w) eps &= a.rec.e_lbl[(size_t)e * 8 + w] == 0u;
        ok = eps && present(i, o, a.rec.e_src[e]);
      }
      const unsigned m = __ballot_sync(0xffffffffu, ok);
      if (m) eps_src = __shfl_sync(0xffffffffu, e < a.in_off[j + 1] ? a.rec.e_src[e] : -1, __ffs(m) - 1);
    }
    if (eps_src >= 0) {
      push(i, o, eps_src, gi);
      continue;
    }
    const int X = g.item_next[i - 1];
    const bool gap = a.rec.col_gap[j] != 0;
    if (X < T) {
      // 2. scanned on a labelled edge, or inside the gap
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
        push(i - 1, o, src, gi);
        continue;
      }
      if (gap && present(i - 1, o, j)) {
        emit(X, true);
        push(i - 1, o, j, gi);
        continue;
      }
      status = 3;
      break;
    }
    const int Bn = X - T;
    // 3a. advanced inside the gap: a shortest string of X
    if (gap && present(i - 1, o, j)) {
      for (int y = g.ny_off[Bn + 1] - 1; y >= g.ny_off[Bn] && status == 0; --y) emit(g.ny[y], true);
      push(i - 1, o, j, gi);
      continue;
    }
    // 3b. a nullable X (the advance over it at j)
    if (!gap && ((g.nullable_next[(i - 1) >> 5] >> ((i - 1) & 31)) & 1u) && present(i - 1, o, j)) {
      push(i - 1, o, j, gi);
      continue;
    }
    // 3c. X completed from m at j, m from j - 1 down to o
    bool found = false;
    for (int mt = j - 1; mt >= o && !found; mt -= 32) {
      const int m = mt - lane;
      const bool ok = m >= o && present(i - 1, o, m) && completes(Bn, m, j);
      unsigned cand = __ballot_sync(0xffffffffu, ok);
      while (cand && !found) {
        const int l = __ffs(cand) - 1;  // lowest lane = highest m
        cand &= cand - 1;
        const int mm = mt - l;
        // a complete item of X at (j, mm), not repeating a same-span ancestor
        const int c0 = g.nt_comp_off[Bn], c1 = g.nt_comp_off[Bn + 1];
        for (int cb = c0; cb < c1 && !found; cb += 32) {
          const int c = cb + lane;
          bool okq = c < c1 && present(g.nt_comp[c], mm, j);
          if (okq && mm == o) {  // same span as this goal: no ancestor with the same item
            int u = gi;
            for (int guard = 0; u >= 0 && guard < 4096; ++guard) {
              if (G[u].item == g.nt_comp[c]) {
                okq = false;
                break;
              }
              u = G[u].up;
            }
          }
          const unsigned qm = __ballot_sync(0xffffffffu, okq);
          if (qm) {
            const int q = __shfl_sync(0xffffffffu, c < c1 ? g.nt_comp[c] : -1, __ffs(qm) - 1);
            push(i - 1, o, mm, gi);  // the left part, derived after X (right to left)
            push(q, mm, j, gi);
            found = true;
          }
        }
      }
    }
    if (!found) {
      status = 3;
      break;
    }
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
#ifdef EPIC_WITNESS_DEBUG
    if (status != 0 && cap >= 12) {  // measurement builds: where the search stopped
      out_len[b] = -10 - status;
      const WGoal cur = G[ns >= 0 && ns < gcap ? S[ns] : 0];
      const int i = cur.item;
      out[0] = i;
      out[1] = cur.o;
      out[2] = cur.j;
      out[3] = i > 0 ? g.item_next[i - 1] : -1;
      out[4] = a.rec.col_gap[cur.j];
      out[5] = len;
      out[6] = ng;
      out[7] = ns;
      out[8] = T;
      out[9] = a.in_off[cur.j + 1] - a.in_off[cur.j];
      out[10] = present(i - 1, cur.o, cur.j) ? 1 : 0;
      out[11] = i > 0 ? (int)((g.nullable_next[(i - 1) >> 5] >> ((i - 1) & 31)) & 1u) : -1;
      if (cap >= 64) {
        // splits m in [o, j): left part present / X completes from m at j
        const int X = i > 0 ? g.item_next[i - 1] : -1;
        int np = 0, nc = 0, p0 = -1, c0 = -1;
        for (int m = cur.o; m < cur.j; ++m) {
          if (present(i - 1, cur.o, m)) {
            ++np;
            p0 = m;
          }
          if (X >= T && completes(X - T, m, cur.j)) {
            ++nc;
            c0 = m;
          }
        }
        out[12] = np;
        out[13] = p0;
        out[14] = nc;
        out[15] = c0;
        out[16] = present(i, cur.o, cur.j) ? 1 : 0;
        // in-edges: source, label words or-ed, item present at the source
        int q = 17;
        for (int e = a.in_off[cur.j]; e < a.in_off[cur.j + 1] && q + 3 <= 60; ++e) {
          uint32_t lo = 0;
          for (int w = 0; w < 8; ++w) lo |= a.rec.e_lbl[(size_t)e * 8 + w];
          out[q++] = a.rec.e_src[e];
          out[q++] = (int)lo;
          out[q++] = present(i, cur.o, a.rec.e_src[e]) ? 1 : 0;
        }
        out[q] = -99;
      }
    }
#endif
  }
}

void launch_witness(int B, cudaStream_t st, const DevGrammar& g, const SeqPack& sp, int32_t* terms, int cap,
                    int32_t* out_len, void* scratch, unsigned long long* stats) {
  // scratch: every sequence's goal records, then every sequence's stack
  const size_t gcap = (size_t)cap * kWitnessGoalsPerTerm;
  WGoal* goals = (WGoal*)scratch;
  int32_t* stack = (int32_t*)(goals + (size_t)B * gcap);
  const int blocks = (B + kWarpsPerCta - 1) / kWarpsPerCta;
  k_witness<<<blocks, 32 * kWarpsPerCta, 0, st>>>(g, B, sp, terms, cap, out_len, goals, stack, stats);
}

size_t witness_goal_bytes(int cap) { return (size_t)cap * kWitnessGoalsPerTerm * (sizeof(WGoal) + sizeof(int32_t)); }

}  // namespace epic

// Earley columns for wide grammars: one CTA closes each column with a
// Gauss-Seidel sweep over its origins (Alg. 3's completion, highest origin
// first), the whole CTA scattering each origin's completions.
//
// Why a descending sweep visits every origin once: completing nonterminal A
// from origin o at column c advances the items of column o that wait on A;
// those items have origins o2 <= o.  So a row with origin o only receives
// from origins >= o, and once every higher origin is closed, row o's only
// remaining source is the entry of column o with origin o itself (the items
// predicted at o).  That self-loop is closed on its own (one warp, row in
// registers) before the completions are scattered, once, over the other
// entries of column o by every warp (entries of one column have distinct
// origins, so no two warps write one row).  Predictions at c only feed row c
// (items predicted at c have origin c), and completions from c at c are the
// nullable / gap advances of every row (Aycock & Horspool; inside a gap
// every symbol derives some terminal string of the trimmed grammar), so
// predictions are made once the lower origins are closed.
//
// Same graph, chart layout, recording and results as EarleyColsT
// (walk.cuh); only the order of the closure differs (the least fixpoint is
// the same).
#pragma once
#include "walk.cuh"
#include "warpwalk.cuh"  // phase timers

namespace epic {

constexpr int kGsMaxWarps = 16;
constexpr long long kGsMaxSteps = 1ll << 22;  // origin visits per column
constexpr long long kGsMaxIdle = 1ll << 24;   // polls of an idle warp per column (warp-parallel sweep)

// Per-warp scratch of the warp-parallel sweep (dynamic shared memory):
// nonterminal words, then the warp's completion mask.
constexpr int kGsWarpScratch = kMaxVW + kMaxW;
__host__ __device__ inline size_t gs_warp_scratch_bytes() { return (size_t)kGsMaxWarps * kGsWarpScratch * 4; }

// The origin sweep of the CTA walks: warp-parallel for item sets of at most
// 64 words, whose columns are short enough for one warp to scatter (on
// clike-512, W = 64: forward charts 22 % faster), the descending block sweep
// for wider ones (random-stress-1024, W = 213: the warp-parallel sweep took
// 20-45 % longer, one warp scattering columns of hundreds of entries);
// EPIC_GS_PARALLEL=0/1 overrides.
inline int gs_parallel_enabled(int W) {
  const char* e = getenv("EPIC_GS_PARALLEL");
  return e ? (atoi(e) != 0) : (W <= 64 ? 1 : 0);
}

// Shared memory of the Gauss-Seidel columns (beside WalkShared).
struct GsShared {
  uint32_t expn[kMaxW];               // items waiting on the current origin's completions
  uint32_t nnew[kMaxVW];              // nonterminals newly completed from the current origin
  uint32_t nstep[kMaxVW];             // of one self-closure round
  uint32_t vset[kMaxVW];              // nonterminals waited on in this column
  uint32_t vdone[kMaxVW];             // ... already predicted
  uint32_t uni[kMaxW];                // union of the column's rows (waited nonterminals)
  int32_t cur_o;
  int32_t flag;
  int32_t labelled;  // the open column has a labelled arrival (else only epsilon ones)
  int32_t busy;      // warp-parallel sweep: warps holding an origin
};

// Grammar tables read by the per-item loops, staged in shared memory:
// item -> next symbol / lhs (int16 [D]) and the W-word masks.
struct GsTables {
  const int16_t* item_next;
  const int16_t* item_lhs;
  const uint32_t* complete;
  const uint32_t* any_nt;
  const uint32_t* any_term;
  const uint32_t* next_any;
  const uint32_t* nullable_next;
  const uint32_t* adv_pow;  // [2][steps][W] (DevGrammar::adv_pow)
};

__host__ __device__ inline size_t gs_tables_bytes(int D, int W, int steps) {
  auto r = [](size_t b) { return (b + 15) & ~(size_t)15; };
  return 2 * r((size_t)D * 2) + 5 * r((size_t)W * 4) + r((size_t)2 * steps * W * 4);
}

// Block: copy the tables into smem (gs_tables_bytes) and point t at them.
__device__ inline void gs_stage_tables(const DevGrammar& g, unsigned char* smem, GsTables& t) {
  unsigned char* p = smem;
  auto put = [&](const void* src, size_t bytes) -> void* {
    void* dst = p;
    const uint16_t* s2 = (const uint16_t*)src;
    uint16_t* d2 = (uint16_t*)dst;
    for (size_t i = threadIdx.x; i < bytes / 2; i += blockDim.x) d2[i] = s2[i];
    p += (bytes + 15) & ~(size_t)15;
    return dst;
  };
  t.item_next = (const int16_t*)put(g.item_next, (size_t)g.D * 2);
  t.item_lhs = (const int16_t*)put(g.item_lhs, (size_t)g.D * 2);
  t.complete = (const uint32_t*)put(g.complete, (size_t)g.W * 4);
  t.any_nt = (const uint32_t*)put(g.any_nt, (size_t)g.W * 4);
  t.any_term = (const uint32_t*)put(g.any_term, (size_t)g.W * 4);
  t.next_any = (const uint32_t*)put(g.next_any, (size_t)g.W * 4);
  t.nullable_next = (const uint32_t*)put(g.nullable_next, (size_t)g.W * 4);
  t.adv_pow = (const uint32_t*)put(g.adv_pow, (size_t)2 * g.adv_steps * g.W * 4);
  __syncthreads();
}

template <bool REC>
class EarleyColsGS {
 public:
  static constexpr int KW = kMaxW / 32;  // item words per lane
  const DevGrammar& g;
  const GsTables& tb;
  const LexEntry* table;
  Workspace ws;
  WalkScratch sc;
  WsDims dims;
  WalkShared& sh;
  GsShared& gs;
  int W, VW;
  static constexpr bool kRecord = REC;
  const BlockRec* rec = nullptr;
  uint32_t* wnt = nullptr;  // recording walks: per-warp nonterminal sets [warps][kMaxVW] (shared memory)
  // Warp-parallel sweep (set both): every warp claims dirty origins on its
  // own and scatters their completions alone; ws.bdone keeps, per origin of
  // the open column, the nonterminals whose completions were scattered.
  bool par = false;
  uint32_t* wscr = nullptr;  // [warps][kGsWarpScratch] (shared memory)

  __device__ EarleyColsGS(const DevGrammar& g_, const GsTables& t_, const LexEntry* t, Workspace w, WalkScratch s,
                          WsDims d, WalkShared& shared, GsShared& gss)
      : g(g_), tb(t_), table(t), ws(w), sc(s), dims(d), sh(shared), gs(gss), W(g_.W), VW(g_.VW) {}

  __device__ int nwarps() const { return blockDim.x >> 5; }
  __device__ bool column_has_accept(int c, int start_col) { return accepts(c, start_col); }
  __device__ void seed(int c) { arrive_item(c, g.start_item); }
  __device__ void arrive_labels(int src, bool eps) { arrive(src, eps ? nullptr : sh.lbl, !eps); }

  __device__ void reset() {
    if (threadIdx.x == 0) {
      sh.ncols = 0;
      sh.nent = 0;
      sh.status = kWalkOk;
      sh.nedges = 0;
      ws.col_off[0] = 0;
    }
    clear_bitmap(sh.touched, kMaxCols);
    clear_bitmap(sh.dirty, kMaxCols);
    for (int v = threadIdx.x; v < kMaxVW; v += blockDim.x) {
      gs.vset[v] = 0;
      gs.vdone[v] = 0;
    }
    if (threadIdx.x == 0) gs.labelled = 0;
    __syncthreads();
  }

  __device__ int ncols() const { return sh.ncols; }
  __device__ int open_column() {
    int c = sh.ncols;
    if (c >= dims.nmax || c >= kMaxCols) {
      if (threadIdx.x == 0) sh.status = kWalkOverflow;
      return -1;
    }
    return c;
  }

  // ------------------------------------------------------------ row kernels
  // Warp: dst |= shift(src & M) (or src & M, or src when M is null), lanes over
  // words; returns whether dst changed.  dst is owned by this warp.
  __device__ bool warp_or_into(uint32_t* dst, const uint32_t* src, const uint32_t* M, bool shift) {
    const int lane = threadIdx.x & 31;
    uint32_t v[KW];
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      const int w = lane + 32 * i;
      v[i] = (w < W) ? (M ? (src[w] & M[w]) : src[w]) : 0u;
    }
    bool ch = false;
    uint32_t carry = 0;
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      if (32 * i >= W) break;
      const int w = lane + 32 * i;
      uint32_t add = v[i];
      if (shift) {
        uint32_t prev = __shfl_up_sync(0xffffffffu, v[i], 1);
        if (lane == 0) prev = carry;
        carry = __shfl_sync(0xffffffffu, v[i], 31);
        add = (v[i] << 1) | (prev >> 31);
      }
      if (w < W && add) {
        const uint32_t old = dst[w];
        if ((old | add) != old) {
          dst[w] = old | add;
          ch = true;
        }
      }
    }
    return __any_sync(0xffffffffu, ch);
  }

  // Warp, row in registers (lane l holds words l, l+32, ...): the closure of r
  // under item i -> i + 1 for i in the advance mask (mode 0: nullable_next,
  // 1: next_any), by doubling: step s adds i + 2^s for every i in r that
  // starts a run of 2^s advanceable items; steps in increasing order reach
  // every i + d with d < 2^steps, which covers the longest production.
  __device__ void reg_advance(uint32_t (&r)[KW], int mode) {
    const int lane = threadIdx.x & 31;
    for (int st = 0; st < g.adv_steps; ++st) {
      const uint32_t* M = tb.adv_pow + ((size_t)mode * g.adv_steps + st) * W;
      const int k = 1 << st;
      if (k < 32) {
        uint32_t carry = 0;
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          if (32 * i >= W) break;
          const int w = lane + 32 * i;
          const uint32_t v = (w < W) ? (r[i] & M[w]) : 0u;
          uint32_t prev = __shfl_up_sync(0xffffffffu, v, 1);
          if (lane == 0) prev = carry;
          carry = __shfl_sync(0xffffffffu, v, 31);
          r[i] |= (v << k) | (prev >> (32 - k));
        }
      } else {  // whole words: word w takes word w - k/32 (never above 64: rhs <= 62)
        const int dw = k >> 5;
        uint32_t v[KW];
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          const int w = lane + 32 * i;
          v[i] = (w < W) ? (r[i] & M[w]) : 0u;
        }
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          if (32 * i >= W) break;
          // source word lane + 32 i - dw, dw in {1, 2}
          const int sl = (lane - dw) & 31;
          const uint32_t same = __shfl_sync(0xffffffffu, v[i], sl);
          const uint32_t prevw = (i > 0) ? __shfl_sync(0xffffffffu, v[i > 0 ? i - 1 : 0], sl) : 0u;
          r[i] |= (lane >= dw) ? same : prevw;
        }
      }
    }
  }

  // Arrivals: for every entry (o, y) of column src, stage[o] |= shift(y & M).
  __device__ void arrive(int src, const uint32_t* M, bool shift) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = nwarps();
    if (shift && threadIdx.x == 0) gs.labelled = 1;
    if (REC && threadIdx.x == 0) {
      if (sh.nedges >= rec->edge_cap) {
        sh.status = kWalkOverflow;
      } else {
        const int e = sh.nedges++;
        rec->e_dst[e] = sh.ncols;
        rec->e_src[e] = src;
        for (int w = 0; w < 8; ++w) rec->e_lbl[(size_t)e * 8 + w] = shift ? sh.lbl8[w] : 0u;
      }
    }
    const int b = ws.col_off[src], e = ws.col_off[src + 1];
    for (int k = b + warp; k < e; k += nw) {
      const int o = ws.org[k];
      const bool ch = warp_or_into(ws.stage + (size_t)o * W, ws.bits + (size_t)k * W, M, shift);
      if (ch && lane == 0) {
        atomicOr(&sh.touched[o >> 5], 1u << (o & 31));
        atomicOr(&sh.dirty[o >> 5], 1u << (o & 31));
      }
    }
    __syncthreads();
  }

  __device__ void arrive_item(int origin, int item) {
    if (threadIdx.x == 0) {
      ws.stage[(size_t)origin * W + (item >> 5)] |= 1u << (item & 31);
      sh.touched[origin >> 5] |= 1u << (origin & 31);
      sh.dirty[origin >> 5] |= 1u << (origin & 31);
    }
    __syncthreads();
  }

  // Warp: highest set bit of bm at or below `top`, or -1.
  __device__ static int warp_highest_at_or_below(const uint32_t* bm, int top) {
    const int lane = threadIdx.x & 31;
    if (top < 0) return -1;
    for (int wtop = top >> 5; wtop >= 0; wtop -= 32) {
      const int w = wtop - lane;
      uint32_t v = (w >= 0) ? bm[w] : 0u;
      if (w == (top >> 5)) v &= (top & 31) == 31 ? 0xffffffffu : ((2u << (top & 31)) - 1u);
      const unsigned any = __ballot_sync(0xffffffffu, v != 0);
      if (any) {
        const int l = __ffs(any) - 1;
        const uint32_t vv = __shfl_sync(0xffffffffu, v, l);
        return ((wtop - l) << 5) + (31 - __clz(vv));
      }
    }
    return -1;
  }

  // Warp 0: close origin o's row on its own (the self-loop through the entry
  // of column o with origin o); leaves the nonterminals newly completed from
  // o in gs.nnew.  Returns whether there are any.
  __device__ bool close_origin(int o, int mode) {
    const int lane = threadIdx.x & 31;
#ifdef EPIC_PHASE_TIMERS
    if (lane == 0) atomicAdd(&g_phase[15], 1ull);
#endif
    uint32_t* row = ws.stage + (size_t)o * W;
    uint32_t r[KW], e[KW];
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      const int w = lane + 32 * i;
      r[i] = (w < W) ? row[w] : 0u;
      e[i] = 0u;
    }
    const int kb = ws.col_off[o], ke = ws.col_off[o + 1];
    const bool self = ke > kb && ws.org[ke - 1] == o;  // entries are stored by ascending origin
    if (self) {
      const uint32_t* E = ws.bits + (size_t)(ke - 1) * W;
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        e[i] = (w < W) ? (E[w] & tb.any_nt[w]) : 0u;
      }
    }
    uint32_t done = 0, tot = 0;  // lane v < VW: word v of the completed / new sets
    uint32_t cseen[KW];          // complete items already counted
#pragma unroll
    for (int i = 0; i < KW; ++i) cseen[i] = 0u;
    for (int round = 0; round < 64 * kMaxW; ++round) {
#ifdef EPIC_PHASE_TIMERS
      if (lane == 0) atomicAdd(&g_phase[14], 1ull);
#endif
      reg_advance(r, mode);
      if (lane < VW) gs.nstep[lane] = 0;
      __syncwarp();
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        uint32_t m = (w < W) ? (r[i] & tb.complete[w] & ~cseen[i]) : 0u;
        cseen[i] |= m;
        while (m) {
          const int b = __ffs(m) - 1;
          m &= m - 1;
          const int A = tb.item_lhs[(w << 5) + b];
          atomicOr(&gs.nstep[A >> 5], 1u << (A & 31));
        }
      }
      __syncwarp();
      const uint32_t nw = (lane < VW) ? (gs.nstep[lane] & ~done) : 0u;
      done |= nw;
      tot |= nw;
      if (!__any_sync(0xffffffffu, nw != 0) || !self) break;
      if (lane < VW) gs.nstep[lane] = nw;
      __syncwarp();
      // the self entry's items waiting on a new nonterminal advance into r
      bool ch = false;
      uint32_t carry = 0;
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        if (32 * i >= W) break;
        const int w = lane + 32 * i;
        uint32_t x = 0, m = e[i];
        while (m) {
          const int b = __ffs(m) - 1;
          m &= m - 1;
          const int B = tb.item_next[(w << 5) + b] - g.T;
          if ((gs.nstep[B >> 5] >> (B & 31)) & 1u) x |= 1u << b;
        }
        uint32_t prev = __shfl_up_sync(0xffffffffu, x, 1);
        if (lane == 0) prev = carry;
        carry = __shfl_sync(0xffffffffu, x, 31);
        const uint32_t add = ((x << 1) | (prev >> 31)) & ~r[i];
        ch |= add != 0;
        r[i] |= add;
      }
      __syncwarp();
      if (!__any_sync(0xffffffffu, ch)) break;
    }
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      const int w = lane + 32 * i;
      if (w < W) row[w] = r[i];
    }
    if (lane < VW) gs.nnew[lane] = tot;
    __syncwarp();
    return __any_sync(0xffffffffu, tot != 0);
  }

  // Block: gs.expn = items waiting on a member of gs.nnew (item test per word).
  __device__ void build_expn() {
    for (int w = threadIdx.x; w < W; w += blockDim.x) {
      uint32_t acc = 0, m = tb.any_nt[w];
      while (m) {
        const int b = __ffs(m) - 1;
        m &= m - 1;
        const int B = tb.item_next[(w << 5) + b] - g.T;
        if ((gs.nnew[B >> 5] >> (B & 31)) & 1u) acc |= 1u << b;
      }
      gs.expn[w] = acc;
    }
  }

  // Block: completions from origin o into the rows of the other entries of
  // column o: stage[org] |= shift(bits & gs.expn).  One thread per (entry,
  // word), consecutive threads on consecutive words (coalesced), four words
  // in flight per thread; entries of one column have distinct origins, so
  // every stage word has one writer.  Changed entries are flagged in
  // gs.chg, then their origins marked touched and dirty.
  __device__ void scatter_column(int o) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = nwarps();
    const int kb = ws.col_off[o], ke = ws.col_off[o + 1];
    const int ne = ke - kb;
    const bool self = ne > 0 && ws.org[ke - 1] == o;
    const int nsc = self ? ne - 1 : ne;  // the self entry is the last one
#ifdef EPIC_PHASE_TIMERS
    if (threadIdx.x == 0) atomicAdd(&g_phase[12], (unsigned long long)nsc * W);
#endif
    // the completion mask in registers: lane l holds words l, l + 32, ...
    uint32_t ex[KW];
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      const int w = lane + 32 * i;
      ex[i] = (w < W) ? gs.expn[w] : 0u;
    }
    const uint32_t* __restrict__ bits = ws.bits + (size_t)kb * W;
    // one warp per entry, two entries in flight; entries of one column have
    // distinct origins, so every stage row has one writer
    for (int e0 = warp; e0 < nsc; e0 += 2 * nw) {
      const int e1 = e0 + nw;
      const bool has1 = e1 < nsc;
      const uint32_t* s0 = bits + (size_t)e0 * W;
      const uint32_t* s1 = bits + (size_t)(has1 ? e1 : e0) * W;
      uint32_t v0[KW], v1[KW];
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        v0[i] = ex[i] ? (__ldg(s0 + w) & ex[i]) : 0u;
        v1[i] = (ex[i] && has1) ? (__ldg(s1 + w) & ex[i]) : 0u;
      }
      uint32_t* d0 = ws.stage + (size_t)ws.org[kb + e0] * W;
      uint32_t* d1 = ws.stage + (size_t)ws.org[kb + (has1 ? e1 : e0)] * W;
      // the shifted words (item (p, d) -> (p, d + 1)), then every destination
      // word loaded before any store (no store may alias a pending load)
      uint32_t a0[KW], a1[KW];
      {
        uint32_t c0 = 0, c1 = 0;
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          uint32_t p0 = __shfl_up_sync(0xffffffffu, v0[i], 1);
          uint32_t p1 = __shfl_up_sync(0xffffffffu, v1[i], 1);
          if (lane == 0) {
            p0 = c0;
            p1 = c1;
          }
          c0 = __shfl_sync(0xffffffffu, v0[i], 31);
          c1 = __shfl_sync(0xffffffffu, v1[i], 31);
          a0[i] = (v0[i] << 1) | (p0 >> 31);
          a1[i] = has1 ? ((v1[i] << 1) | (p1 >> 31)) : 0u;
        }
      }
      uint32_t q0[KW], q1[KW];
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        q0[i] = (w < W && a0[i]) ? d0[w] : 0u;
        q1[i] = (w < W && a1[i]) ? d1[w] : 0u;
      }
      bool ch0 = false, ch1 = false;
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        if (w < W && (a0[i] & ~q0[i])) {
          d0[w] = q0[i] | a0[i];
          ch0 = true;
        }
        if (w < W && (a1[i] & ~q1[i])) {
          d1[w] = q1[i] | a1[i];
          ch1 = true;
        }
      }
      ch0 = __any_sync(0xffffffffu, ch0);
      ch1 = __any_sync(0xffffffffu, ch1);
      if (lane == 0) {
        if (ch0) {
          const int o2 = ws.org[kb + e0];
          atomicOr(&sh.touched[o2 >> 5], 1u << (o2 & 31));
          atomicOr(&sh.dirty[o2 >> 5], 1u << (o2 & 31));
        }
        if (ch1 && has1) {
          const int o2 = ws.org[kb + e1];
          atomicOr(&sh.touched[o2 >> 5], 1u << (o2 & 31));
          atomicOr(&sh.dirty[o2 >> 5], 1u << (o2 & 31));
        }
      }
    }
    __syncthreads();
  }

  // ------------------------------------------------------ warp-parallel sweep
  // The same least fixpoint as the descending sweep, reached without block
  // barriers: each warp repeatedly claims the highest dirty origin below c
  // (clearing its bit), closes its row with the self-loop, claims in
  // ws.bdone the nonterminals it completes that no visit scattered yet, and
  // scatters those over column o with atomic ORs, marking the rows it changes
  // dirty again.  A row may be claimed while another warp still writes into
  // it; the writer sets the dirty bit after its writes (fenced), so the row
  // is visited again and nothing is lost.  The sweep ends when no bit is
  // dirty and no warp holds an origin.  Rows are read through L2 (ld.cg):
  // other warps' atomics do not update this SM's L1.

  __device__ static int warp_highest_dirty(const uint32_t* bm, int top) {
    const int lane = threadIdx.x & 31;
    if (top < 0) return -1;
    const volatile uint32_t* vb = bm;
    for (int wtop = top >> 5; wtop >= 0; wtop -= 32) {
      const int w = wtop - lane;
      uint32_t v = (w >= 0) ? vb[w] : 0u;
      if (w == (top >> 5)) v &= (top & 31) == 31 ? 0xffffffffu : ((2u << (top & 31)) - 1u);
      const unsigned any = __ballot_sync(0xffffffffu, v != 0);
      if (any) {
        const int l = __ffs(any) - 1;
        const uint32_t vv = __shfl_sync(0xffffffffu, v, l);
        return ((wtop - l) << 5) + (31 - __clz(vv));
      }
    }
    return -1;
  }

  // Warp: close row o with its self-loop (as close_origin), the nonterminals
  // already scattered for o taken as done; returns, in lane v < VW, word v of
  // the nonterminals this visit claimed (completed from o and not yet
  // scattered by any visit).
  __device__ uint32_t close_origin_claim(int o, int mode, uint32_t* nstep) {
    const int lane = threadIdx.x & 31;
    uint32_t* row = ws.stage + (size_t)o * W;
    uint32_t* bd = ws.bdone + (size_t)o * VW;
    // done before the row: a visit writes its row before it claims
    uint32_t known = (lane < VW) ? __ldcg(bd + lane) : 0u;
    __threadfence_block();
    uint32_t r[KW], r0[KW], e[KW];
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      const int w = lane + 32 * i;
      r[i] = (w < W) ? __ldcg(row + w) : 0u;
      r0[i] = r[i];
      e[i] = 0u;
    }
    const int kb = ws.col_off[o], ke = ws.col_off[o + 1];
    const bool self = ke > kb && ws.org[ke - 1] == o;
    if (self) {
      const uint32_t* E = ws.bits + (size_t)(ke - 1) * W;
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        e[i] = (w < W) ? (E[w] & tb.any_nt[w]) : 0u;
      }
    }
    uint32_t tot = 0;
    uint32_t cseen[KW];
#pragma unroll
    for (int i = 0; i < KW; ++i) cseen[i] = 0u;
    for (int round = 0; round < 64 * kMaxW; ++round) {
      reg_advance(r, mode);
      if (lane < VW) nstep[lane] = 0;
      __syncwarp();
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        uint32_t m = (w < W) ? (r[i] & tb.complete[w] & ~cseen[i]) : 0u;
        cseen[i] |= m;
        while (m) {
          const int b = __ffs(m) - 1;
          m &= m - 1;
          const int A = tb.item_lhs[(w << 5) + b];
          atomicOr(&nstep[A >> 5], 1u << (A & 31));
        }
      }
      __syncwarp();
      const uint32_t nw = (lane < VW) ? (nstep[lane] & ~known) : 0u;
      known |= nw;
      tot |= nw;
      if (!__any_sync(0xffffffffu, nw != 0) || !self) break;
      if (lane < VW) nstep[lane] = nw;
      __syncwarp();
      bool ch = false;
      uint32_t carry = 0;
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        if (32 * i >= W) break;
        const int w = lane + 32 * i;
        uint32_t x = 0, m = e[i];
        while (m) {
          const int b = __ffs(m) - 1;
          m &= m - 1;
          const int B = tb.item_next[(w << 5) + b] - g.T;
          if ((nstep[B >> 5] >> (B & 31)) & 1u) x |= 1u << b;
        }
        uint32_t prev = __shfl_up_sync(0xffffffffu, x, 1);
        if (lane == 0) prev = carry;
        carry = __shfl_sync(0xffffffffu, x, 31);
        const uint32_t add = ((x << 1) | (prev >> 31)) & ~r[i];
        ch |= add != 0;
        r[i] |= add;
      }
      __syncwarp();
      if (!__any_sync(0xffffffffu, ch)) break;
    }
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      const int w = lane + 32 * i;
      if (w < W && (r[i] & ~r0[i])) atomicOr(row + w, r[i]);
    }
    __threadfence_block();
    uint32_t mine = 0;
    if (lane < VW && tot) mine = tot & ~atomicOr(bd + lane, tot);
    return mine;
  }

  // Warp: completions of the nonterminals in nnew (nnew[v], v < VW) from
  // origin o into the rows of the other entries of column o.
  __device__ void scatter_warp(int o, const uint32_t* nnew, uint32_t* expn) {
    const int lane = threadIdx.x & 31;
    for (int w = lane; w < W; w += 32) {
      uint32_t acc = 0, m = tb.any_nt[w];
      while (m) {
        const int b = __ffs(m) - 1;
        m &= m - 1;
        const int B = tb.item_next[(w << 5) + b] - g.T;
        if ((nnew[B >> 5] >> (B & 31)) & 1u) acc |= 1u << b;
      }
      expn[w] = acc;
    }
    __syncwarp();
    uint32_t ex[KW];
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      const int w = lane + 32 * i;
      ex[i] = (w < W) ? expn[w] : 0u;
    }
    const int kb = ws.col_off[o], ke = ws.col_off[o + 1];
    const bool self = ke > kb && ws.org[ke - 1] == o;
    const int nsc = (self ? ke - 1 : ke) - kb;
    const uint32_t* __restrict__ bits = ws.bits + (size_t)kb * W;
    for (int e0 = 0; e0 < nsc; e0 += 2) {
      const bool has1 = e0 + 1 < nsc;
      const uint32_t* s0 = bits + (size_t)e0 * W;
      const uint32_t* s1 = bits + (size_t)(has1 ? e0 + 1 : e0) * W;
      uint32_t v0[KW], v1[KW];
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        v0[i] = ex[i] ? (__ldg(s0 + w) & ex[i]) : 0u;
        v1[i] = (ex[i] && has1) ? (__ldg(s1 + w) & ex[i]) : 0u;
      }
      const int o0 = ws.org[kb + e0], o1 = ws.org[kb + (has1 ? e0 + 1 : e0)];
      uint32_t* d0 = ws.stage + (size_t)o0 * W;
      uint32_t* d1 = ws.stage + (size_t)o1 * W;
      uint32_t a0[KW], a1[KW];
      {
        uint32_t c0 = 0, c1 = 0;
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          uint32_t p0 = __shfl_up_sync(0xffffffffu, v0[i], 1);
          uint32_t p1 = __shfl_up_sync(0xffffffffu, v1[i], 1);
          if (lane == 0) {
            p0 = c0;
            p1 = c1;
          }
          c0 = __shfl_sync(0xffffffffu, v0[i], 31);
          c1 = __shfl_sync(0xffffffffu, v1[i], 31);
          a0[i] = (v0[i] << 1) | (p0 >> 31);
          a1[i] = has1 ? ((v1[i] << 1) | (p1 >> 31)) : 0u;
        }
      }
      uint32_t q0[KW], q1[KW];
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        q0[i] = (w < W && a0[i]) ? __ldcg(d0 + w) : 0u;
        q1[i] = (w < W && a1[i]) ? __ldcg(d1 + w) : 0u;
      }
      bool ch0 = false, ch1 = false;
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        if (w < W && (a0[i] & ~q0[i])) {
          atomicOr(d0 + w, a0[i]);
          ch0 = true;
        }
        if (w < W && (a1[i] & ~q1[i])) {
          atomicOr(d1 + w, a1[i]);
          ch1 = true;
        }
      }
      __threadfence_block();  // every lane's row writes before the dirty bits
      ch0 = __any_sync(0xffffffffu, ch0);
      ch1 = __any_sync(0xffffffffu, ch1);
      __syncwarp();
      if (lane == 0) {
        if (ch0) {
          atomicOr(&sh.touched[o0 >> 5], 1u << (o0 & 31));
          atomicOr(&sh.dirty[o0 >> 5], 1u << (o0 & 31));
        }
        if (ch1 && has1) {
          atomicOr(&sh.touched[o1 >> 5], 1u << (o1 & 31));
          atomicOr(&sh.dirty[o1 >> 5], 1u << (o1 & 31));
        }
      }
      __syncwarp();
    }
  }

  // Block: the origins below c, closed warp-parallel (every warp returns
  // when the sweep is done).
  __device__ void close_origins_par(int c, int mode) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint32_t* nstep = wscr + (size_t)warp * kGsWarpScratch;
    uint32_t* expn = nstep + kMaxVW;
    volatile int32_t* busy = &gs.busy;
    long long visits = 0, idle = 0;
    for (;;) {
      // claim the highest dirty origin; a holder counts itself busy right
      // after its claim (a warp that saw nothing dirty and no holder in that
      // gap leaves early, and the holder finishes what its origin causes)
      int o = -1;
      for (int tries = 0; tries < 64; ++tries) {
        const int h = warp_highest_dirty(sh.dirty, c - 1);
        if (h < 0) break;
        uint32_t old = 0;
        if (lane == 0) {
          old = atomicAnd(&sh.dirty[h >> 5], ~(1u << (h & 31)));
          if ((old >> (h & 31)) & 1u) atomicAdd(&gs.busy, 1);
        }
        old = __shfl_sync(0xffffffffu, old, 0);
        if ((old >> (h & 31)) & 1u) {
          o = h;
          break;
        }
      }
      if (o < 0) {
        // done when no warp holds an origin and, after that, nothing is dirty
        int b = 0;
        if (lane == 0) b = *busy;
        b = __shfl_sync(0xffffffffu, b, 0);
        __threadfence_block();
        if (b == 0 && warp_highest_dirty(sh.dirty, c - 1) < 0) break;
        if (++idle > kGsMaxIdle) {
          if (lane == 0) sh.status = kWalkOverflow;
          break;
        }
        __nanosleep(64);
        continue;
      }
      __syncwarp();  // the claim (lane 0) before any lane reads the row
      __threadfence_block();
      if (++visits > kGsMaxSteps) {
        if (lane == 0) {
          sh.status = kWalkOverflow;
          atomicSub(&gs.busy, 1);
        }
        __syncwarp();
        break;
      }
      const uint32_t mine = close_origin_claim(o, mode, nstep);
      if (lane < VW) nstep[lane] = mine;
      __syncwarp();
      if (__any_sync(0xffffffffu, mine != 0)) scatter_warp(o, nstep, expn);
      __threadfence_block();
      __syncwarp();
      if (lane == 0) atomicSub(&gs.busy, 1);
      __syncwarp();
    }
  }

  // Closure of column c (gap: a node with a Sigma_lex* self-loop).
  __device__ void close_column(int c, bool gap) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = nwarps();
    if (REC && threadIdx.x == 0) rec->col_gap[c] = gap ? 1 : 0;
    const int mode = gap ? 1 : 0;  // the advance rule: next_any in a gap, nullable_next elsewhere
    // 1. origins below c, highest first; warp 0 walks down the dirty origins
    //    until one completes something new, then every warp scatters.
    //    A node (not a gap) reached only by epsilon edges from finished
    //    columns needs none of it: each of its rows is a union of rows that
    //    are closed under completion and advance, and so is the union (what
    //    an origin completes here, it completed in one of the sources, whose
    //    rows below already hold the advanced items).
    int top = (!gap && !gs.labelled) ? -1 : c - 1;
    if (par) {
      if (threadIdx.x == 0) gs.busy = 0;
      __syncthreads();
      if (top >= 0) close_origins_par(c, mode);
      __syncthreads();
      if (sh.status == kWalkOverflow) return;
      top = -1;  // the descending sweep below has nothing left
    }
    for (long long step = 0;; ++step) {
      if (warp == 0) {
        PH_BEGIN(t_or);
        int o = -1;
        for (long long guard = 0; guard <= kGsMaxSteps; ++guard) {
          o = warp_highest_at_or_below(sh.dirty, top);
          if (o < 0) break;
          if (lane == 0) sh.dirty[o >> 5] &= ~(1u << (o & 31));
          __syncwarp();
          top = o - 1;
          if (close_origin(o, mode)) break;
          o = -1;
        }
        if (lane == 0) gs.cur_o = o;
        PH_END(8, t_or);
      }
      __syncthreads();
      const int o = gs.cur_o;
      if (o < 0) break;
      if (step > kGsMaxSteps) {
        if (threadIdx.x == 0) sh.status = kWalkOverflow;
        __syncthreads();
        return;
      }
      PH_BEGIN(t_sc);
      build_expn();
      __syncthreads();
      scatter_column(o);
      PH_END(9, t_sc);
    }
    // 2. predictions: nonterminals waited on by any row of the column; row c
    //    is closed with them (its completions at c are the advance rules)
    PH_BEGIN(t_pr);
    for (int w = threadIdx.x; w < W; w += blockDim.x) gs.uni[w] = 0;
    __syncthreads();
    bitmap_to_list(sh, sh.touched, c + 1);
    const int nl = sh.list_n;
    for (int i = warp; i < nl; i += nw) {
      const uint32_t* row = ws.stage + (size_t)sh.list[i] * W;
      for (int w = lane; w < W; w += 32) {
        const uint32_t v = row[w] & tb.any_nt[w];
        if (v) atomicOr(&gs.uni[w], v);
      }
    }
    __syncthreads();
    for (int round = 0; round < 4 * kMaxVW + 4; ++round) {
      // vset |= nonterminals after the dot in uni
      for (int w = threadIdx.x; w < W; w += blockDim.x) {
        uint32_t m = gs.uni[w];
        while (m) {
          const int b = __ffs(m) - 1;
          m &= m - 1;
          const int B = tb.item_next[(w << 5) + b] - g.T;
          atomicOr(&gs.vset[B >> 5], 1u << (B & 31));
        }
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        uint32_t any = 0;
        for (int v = 0; v < VW; ++v) {
          const uint32_t nw2 = gs.vset[v] & ~gs.vdone[v];
          gs.nnew[v] = nw2;
          any |= nw2;
        }
        gs.flag = any != 0;
      }
      __syncthreads();
      if (!gs.flag) break;
      const uint32_t* P = gap ? g.gap_pred : g.pred;
      uint32_t* crow = ws.stage + (size_t)c * W;
      for (int w = threadIdx.x; w < W; w += blockDim.x) {
        uint32_t acc = 0;
        for (int v = 0; v < VW; ++v) {
          uint32_t m = gs.nnew[v];
          while (m) {
            const int b = __ffs(m) - 1;
            m &= m - 1;
            acc |= P[(size_t)((v << 5) + b) * W + w];
          }
        }
        crow[w] |= acc;
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        for (int v = 0; v < VW; ++v) gs.vdone[v] |= gs.nnew[v];
        sh.touched[c >> 5] |= 1u << (c & 31);
      }
      if (warp == 0) {  // advance row c, add its items to uni
        uint32_t r[KW];
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          const int w = lane + 32 * i;
          r[i] = (w < W) ? crow[w] : 0u;
        }
        reg_advance(r, mode);
#pragma unroll
        for (int i = 0; i < KW; ++i) {
          const int w = lane + 32 * i;
          if (w < W) {
            crow[w] = r[i];
            gs.uni[w] |= r[i] & tb.any_nt[w];
          }
        }
      }
      __syncthreads();
    }
    // a seeded row c (the walk's first column) is closed by the advance as well
    if (warp == 0 && bit_get(sh.dirty, c)) {
      uint32_t* crow = ws.stage + (size_t)c * W;
      uint32_t r[KW];
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        r[i] = (w < W) ? crow[w] : 0u;
      }
      reg_advance(r, mode);
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        const int w = lane + 32 * i;
        if (w < W) crow[w] = r[i];
      }
      if (lane == 0) sh.dirty[c >> 5] &= ~(1u << (c & 31));
    }
    __syncthreads();
    PH_END(10, t_pr);
  }

  // Move the touched nonzero rows into the entry store as column c (origins
  // ascending), recording completed nonterminals and summaries.
  __device__ void finish_column(int c) {
    PH_BEGIN(t_fi);
    finish_inner(c);
    PH_END(11, t_fi);
  }
  __device__ void finish_inner(int c) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = nwarps();
    bitmap_to_list(sh, sh.touched, c + 1);
    const int nl = sh.list_n;
    for (int i = warp; i < nl; i += nw) {
      const uint32_t* row = ws.stage + (size_t)sh.list[i] * W;
      bool nz = false;
      for (int w = lane; w < W; w += 32) nz |= row[w] != 0;
      nz = __any_sync(0xffffffffu, nz);
      if (lane == 0) sh.prefix[i] = nz ? 1 : 0;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int s = 0;
      for (int i = 0; i < nl; ++i) {
        const int f = sh.prefix[i];
        sh.prefix[i] = f ? s : -1;
        s += f;
      }
      const long long base = ws.col_off[c];
      if (base + s > dims.emax) {
        sh.status = kWalkOverflow;
      } else {
        ws.col_off[c + 1] = (int)(base + s);
        sh.nent = base + s;
      }
      sh.ncols = c + 1;
    }
    __syncthreads();
    const bool ok = sh.status != kWalkOverflow;
    const int base = ws.col_off[c];
    for (int i = warp; i < nl; i += nw) {
      const int o = sh.list[i];
      uint32_t* row = ws.stage + (size_t)o * W;
      const int slot = sh.prefix[i];
      if (ok && slot >= 0) {
        if (lane == 0) ws.org[base + slot] = o;
        uint32_t* dst = ws.bits + (size_t)(base + slot) * W;
        for (int w = lane; w < W; w += 32) dst[w] = row[w];
        if constexpr (REC) record_entry(row, (long long)base + slot);
      }
      __syncwarp();
      for (int w = lane; w < W; w += 32) row[w] = 0;
      if (par)
        for (int v = lane; v < VW; v += 32) ws.bdone[(size_t)o * VW + v] = 0;
    }
    clear_bitmap(sh.touched, c + 1);
    clear_bitmap(sh.dirty, c + 1);
    for (int v = threadIdx.x; v < kMaxVW; v += blockDim.x) {
      gs.vset[v] = 0;
      gs.vdone[v] = 0;
    }
    if (threadIdx.x == 0) gs.labelled = 0;
    __syncthreads();
  }

  __device__ bool column_empty(int c) const { return ws.col_off[c + 1] == ws.col_off[c]; }

  // Warp: completed nonterminals and folded summaries of stored entry k.
  __device__ void record_entry(const uint32_t* row, long long k) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint32_t* nts = wnt + (size_t)warp * kMaxVW;
    for (int v = lane; v < VW; v += 32) nts[v] = 0;
    __syncwarp();
    uint32_t fnt = 0, ft = 0;
    for (int w = lane; w < W; w += 32) {
      const uint32_t r = row[w];
      uint32_t m = r & tb.complete[w];
      while (m) {
        const int b = __ffs(m) - 1;
        m &= m - 1;
        const int B = tb.item_lhs[(w << 5) + b];
        atomicOr(&nts[B >> 5], 1u << (B & 31));
      }
      m = r & tb.any_nt[w];
      while (m) {
        const int b = __ffs(m) - 1;
        m &= m - 1;
        fnt |= 1u << ((tb.item_next[(w << 5) + b] - g.T) & 31);
      }
      m = r & tb.any_term[w];
      while (m) {
        const int b = __ffs(m) - 1;
        m &= m - 1;
        ft |= 1u << (tb.item_next[(w << 5) + b] & 31);
      }
    }
    for (int off = 16; off; off >>= 1) {
      fnt |= __shfl_xor_sync(0xffffffffu, fnt, off);
      ft |= __shfl_xor_sync(0xffffffffu, ft, off);
    }
    __syncwarp();
    for (int v = lane; v < VW; v += 32) rec->cnt[(size_t)k * VW + v] = nts[v];
    if (lane == 0) {
      rec->esum[(size_t)k * 2] = fnt;
      rec->esum[(size_t)k * 2 + 1] = ft;
    }
    __syncwarp();
  }

  // After an aborted walk: return the staging rows of the open column to zero.
  __device__ void cleanup() {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = nwarps();
    bitmap_to_list(sh, sh.touched, kMaxCols);
    const int nl = sh.list_n;
    for (int i = warp; i < nl; i += nw) {
      const int o = sh.list[i];
      for (int w = lane; w < W; w += 32) ws.stage[(size_t)o * W + w] = 0;
      if (par)
        for (int v = lane; v < VW; v += 32) ws.bdone[(size_t)o * VW + v] = 0;
    }
    clear_bitmap(sh.touched, kMaxCols);
    clear_bitmap(sh.dirty, kMaxCols);
    for (int v = threadIdx.x; v < kMaxVW; v += blockDim.x) {
      gs.vset[v] = 0;
      gs.vdone[v] = 0;
    }
    if (threadIdx.x == 0) gs.labelled = 0;
    __syncthreads();
  }

  __device__ bool accepts(int c, int start_col) {
    __shared__ int found;
    if (threadIdx.x == 0) found = 0;
    __syncthreads();
    for (int k = ws.col_off[c] + threadIdx.x; k < ws.col_off[c + 1]; k += blockDim.x)
      if (ws.org[k] == start_col && bit_get(ws.bits + (size_t)k * W, g.accept_item)) found = 1;
    __syncthreads();
    return found != 0;
  }
};

}  // namespace epic

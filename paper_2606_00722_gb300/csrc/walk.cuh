// Block-wide Earley recognition over the lexeme graph of a partial output
// (Alg. 3 on the graph of Alg. 2), built on the fly from the lex table.
//
// The graph (the gap reading): every maximal run of masks is a gap node with a
// self-loop on every terminal; every maximal run of tokens is a span whose
// lexings are paths.  Inside a span the graph nodes are (token boundary,
// lexer state) pairs -- lexings that reach the same lexer state at the same
// token boundary continue identically, so they share the node -- plus one
// node per distinct (target, remaining run) between boundaries, so that runs
// that differ only in their first terminal share the rest of their path.
// The paths between two nodes spell exactly the distinct terminal runs of the
// span from its entry states (q0 at the sequence start, every lexer state
// after a gap), flushed at END; so the language of the graph, and hence the
// validity bit, is that of the per-alternative graph of the definition.
//
// Chart (Alg. 3 items): for every graph node c, a list of entries (origin
// node o, bitset over dotted items) -- the items (p, d, o) present at c.
// Predict / scan / complete are bit-parallel: a scan over terminal a is
// ((bits & EXP_T[a]) << 1) because item (p, d+1) follows item (p, d); a
// completion of the nonterminals Bset from origin o' advances the items
// of column o' that wait on a member of Bset; prediction ORs precomputed
// prediction closures; nullable nonterminals are skipped on prediction
// (Aycock & Horspool); inside a gap every item advances over any symbol.
#pragma once
#include "device.cuh"

namespace epic {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxCols = 4096;   // columns (graph nodes) per walk
constexpr int kMaxQ = 1024;      // lexer states
constexpr int kMaxW = 256;       // item words (D <= 8192)
constexpr int kMaxVW = 32;       // nonterminal words (V <= 1024)
constexpr int kMaxRounds = 1 << 14;

enum WalkStatus { kWalkOk = 0, kWalkOverflow = 1, kWalkBadInput = 2, kWalkDead = 3 };

struct Subst {   // (position, token) substitutions, sorted by position
  const int32_t* pos;
  const int32_t* tok;
  int n;
};

// Per-walk global scratch beyond Workspace (group tables of the span step).
struct WalkScratch {
  int32_t* g_src;     // [kMaxQ] group source column
  int32_t* g_end;     // [kMaxQ] group end lexer state
  int32_t* g_len;     // [kMaxQ]
  uint8_t* g_tail;    // [kMaxQ][16] terminals after the first
  uint32_t* g_lbl;    // [kMaxQ][8] first-terminal label set
  int32_t* g_last;    // [kMaxQ] column holding the run before its last terminal
  int32_t* f_q;       // [kMaxQ] frontier lexer states
  int32_t* f_c;       // [kMaxQ] frontier columns
  int32_t* key_q;     // [kMaxQ] member -> leader
  uint32_t* expn;     // [kMaxCols][W] completion masks of the propagating origins
  uint32_t* bnew;     // [kMaxCols][VW]
};

struct WalkShared {
  uint32_t touched[kMaxCols / 32];
  uint32_t dirty[kMaxCols / 32];
  uint32_t next_dirty[kMaxCols / 32];
  uint32_t prop[kMaxCols / 32];
  int32_t list[kMaxCols];
  int32_t list_n;
  int32_t prefix[kMaxCols + 1];
  uint32_t vset[kMaxVW];
  uint32_t vdone[kMaxVW];
  uint32_t lbl[kMaxW];
  uint32_t wnt[kWarps][kMaxVW];
  int32_t ncols;
  long long nent;
  int32_t status;
  int32_t changed;
  int32_t nf, ng, nt;
  int32_t start_col, accept_col;
  int32_t nedges;    // edges recorded so far (recording walks)
  uint32_t lbl8[8];  // terminal set of the arrivals being made
  int32_t scratch_i[4];
};

__device__ __forceinline__ bool bit_get(const uint32_t* m, int i) { return (m[i >> 5] >> (i & 31)) & 1u; }

// ------------------------------------------------------------ block helpers
// Compact the set bits of bitmap[0 .. nbits) into sh.list (ascending).
__device__ inline void bitmap_to_list(WalkShared& sh, const uint32_t* bitmap, int nbits) {
  int nw = (nbits + 31) >> 5;
  for (int w = threadIdx.x; w < nw; w += blockDim.x) sh.prefix[w] = __popc(bitmap[w]);
  __syncthreads();
  if (threadIdx.x == 0) {
    int s = 0;
    for (int w = 0; w < nw; ++w) {
      int c = sh.prefix[w];
      sh.prefix[w] = s;
      s += c;
    }
    sh.list_n = s;
  }
  __syncthreads();
  for (int w = threadIdx.x; w < nw; w += blockDim.x) {
    uint32_t m = bitmap[w];
    int o = sh.prefix[w];
    while (m) {
      int b = __ffs(m) - 1;
      m &= m - 1;
      sh.list[o++] = (w << 5) + b;
    }
  }
  __syncthreads();
}

__device__ __forceinline__ void clear_bitmap(uint32_t* bm, int nbits) {
  for (int w = threadIdx.x; w < ((nbits + 31) >> 5); w += blockDim.x) bm[w] = 0;
}

// Warp: row |= shift(row & M) for a W-word row, until stable; returns true if
// anything changed.  Item (p, d) is bit i, (p, d+1) is bit i+1.
__device__ inline bool warp_advance_closure(uint32_t* row, const uint32_t* M, int W) {
  int lane = threadIdx.x & 31;
  bool any = false;
  for (int it = 0; it < 64; ++it) {
    bool ch = false;
    uint32_t carry = 0;  // (row & M) >> 31 of the previous word
    for (int base = 0; base < W; base += 32) {
      int w = base + lane;
      uint32_t v = (w < W) ? (row[w] & M[w]) : 0u;
      uint32_t prev = __shfl_up_sync(0xffffffffu, v, 1);
      if (lane == 0) prev = carry;
      uint32_t add = (v << 1) | (prev >> 31);
      carry = __shfl_sync(0xffffffffu, v, 31);
      if (w < W) {
        uint32_t old = row[w];
        if ((old | add) != old) {
          row[w] = old | add;
          ch = true;
        }
      }
    }
    __syncwarp();
    ch = __any_sync(0xffffffffu, ch);
    if (!ch) break;
    any = true;
  }
  return any;
}

// Warp: out |= shift(in & M) into the stage row of origin o (atomic OR); returns
// whether anything was nonzero.
__device__ __forceinline__ bool warp_scan_into(uint32_t* dst, const uint32_t* in, const uint32_t* M, int W,
                                               bool shift, bool atomic) {
  int lane = threadIdx.x & 31;
  bool nz = false;
  uint32_t carry = 0;
  for (int base = 0; base < W; base += 32) {
    int w = base + lane;
    uint32_t v = (w < W) ? (M ? (in[w] & M[w]) : in[w]) : 0u;
    uint32_t add = v;
    if (shift) {
      uint32_t prev = __shfl_up_sync(0xffffffffu, v, 1);
      if (lane == 0) prev = carry;
      add = (v << 1) | (prev >> 31);
      carry = __shfl_sync(0xffffffffu, v, 31);
    }
    if (w < W && add) {
      nz = true;
      if (atomic)
        atomicOr(&dst[w], add);
      else
        dst[w] |= add;
    }
  }
  return __any_sync(0xffffffffu, nz);
}

// What a recording walk (a sequence's forward chart, for checks by region)
// writes besides the chart: the graph's edges in target order with their
// terminal sets (all zero: epsilon), gap flags, each entry's completed
// nonterminals and folded summaries (bit B mod 32 of a waited-on nonterminal,
// bit a mod 32 of an expected terminal), and the column before, at and after
// each position's segment.
struct BlockRec {
  uint8_t* col_gap;   // [nmax]
  int32_t* e_dst;     // [edge_cap]
  int32_t* e_src;     // [edge_cap]
  uint32_t* e_lbl;    // [edge_cap][8]
  uint32_t* cnt;      // [emax][VW]
  uint32_t* esum;     // [emax][2]
  int32_t* gap_col;   // [n]
  int32_t* pre_col;   // [n]
  int32_t* post_col;  // [n]
  int edge_cap;
};

// ------------------------------------------------------------ Earley columns
// REC = true: a recording walk (BlockRec), compiled out of the others.
template <bool REC>
class EarleyColsT {
 public:
  const DevGrammar& g;
  const LexEntry* table;
  Workspace ws;
  WalkScratch sc;
  WsDims dims;
  WalkShared& sh;
  int W, VW;
  static constexpr bool kRecord = REC;
  const BlockRec* rec = nullptr;  // recording walks only

  __device__ EarleyColsT(const DevGrammar& g_, const LexEntry* t, Workspace w, WalkScratch s, WsDims d,
                    WalkShared& shared)
      : g(g_), table(t), ws(w), sc(s), dims(d), sh(shared), W(g_.W), VW(g_.VW) {}
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
    clear_bitmap(sh.next_dirty, kMaxCols);
    clear_bitmap(sh.prop, kMaxCols);
    __syncthreads();
  }

  __device__ int ncols() const { return sh.ncols; }
  __device__ int entries_begin(int c) const { return ws.col_off[c]; }
  __device__ int entries_end(int c) const { return ws.col_off[c + 1]; }

  // Open column c = ncols (caller syncs afterwards).
  __device__ int open_column() {
    int c = sh.ncols;
    if (c >= dims.nmax || c >= kMaxCols) {
      if (threadIdx.x == 0) sh.status = kWalkOverflow;
      return -1;
    }
    return c;
  }

  // Arrivals: for every entry (o, y) of column src, stage[o] |= shift(y & M)
  // (M == nullptr and shift == false for an epsilon edge).
  __device__ void arrive(int src, const uint32_t* M, bool shift) {
    int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (REC && threadIdx.x == 0) {  // the edge src -> open column
      if (sh.nedges >= rec->edge_cap) {
        sh.status = kWalkOverflow;
      } else {
        const int e = sh.nedges++;
        rec->e_dst[e] = sh.ncols;
        rec->e_src[e] = src;
        for (int w = 0; w < 8; ++w) rec->e_lbl[(size_t)e * 8 + w] = shift ? sh.lbl8[w] : 0u;
      }
    }
    int b = ws.col_off[src], e = ws.col_off[src + 1];
    for (int k = b + warp; k < e; k += kWarps) {
      int o = ws.org[k];
      bool nz = warp_scan_into(ws.stage + (size_t)o * W, ws.bits + (size_t)k * W, M, W, shift, false);
      if (nz && lane == 0) {
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

  // Closure of column c (is_gap: a gap node with a Sigma_lex* self-loop).
  __device__ void close_column(int c, bool gap) {
    int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (REC && threadIdx.x == 0) rec->col_gap[c] = gap ? 1 : 0;
    for (int round = 0;; ++round) {
      if (round >= kMaxRounds) {
        if (threadIdx.x == 0) sh.status = kWalkOverflow;
        __syncthreads();
        return;
      }
      // A: per dirty origin -- in-row closures, completed and waited-on NTs
      bitmap_to_list(sh, sh.dirty, c + 1);
      if (sh.list_n == 0) break;
      int nl = sh.list_n;
      for (int i = warp; i < nl; i += kWarps) {
        int o = sh.list[i];
        uint32_t* row = ws.stage + (size_t)o * W;
        if (gap) warp_advance_closure(row, g.next_any, W);
        warp_advance_closure(row, g.nullable_next, W);
        for (int v = lane; v < VW; v += 32) sh.wnt[warp][v] = 0;
        __syncwarp();
        for (int w = lane; w < W; w += 32) {
          uint32_t r = row[w];
          uint32_t m = r & g.complete[w];
          while (m) {
            int b = __ffs(m) - 1;
            m &= m - 1;
            int B = g.item_lhs[(w << 5) + b];
            atomicOr(&sh.wnt[warp][B >> 5], 1u << (B & 31));
          }
          m = r & g.any_nt[w];
          while (m) {
            int b = __ffs(m) - 1;
            m &= m - 1;
            int B = g.item_next[(w << 5) + b] - g.T;
            atomicOr(&sh.vset[B >> 5], 1u << (B & 31));
          }
        }
        __syncwarp();
        if (o != c) {
          bool any = false;
          for (int v = lane; v < VW; v += 32) {
            uint32_t done = ws.bdone[(size_t)o * VW + v];
            uint32_t nw = sh.wnt[warp][v] & ~done;
            sc.bnew[(size_t)o * VW + v] = nw;
            if (nw) any = true;
          }
          any = __any_sync(0xffffffffu, any);
          if (any && lane == 0) atomicOr(&sh.prop[o >> 5], 1u << (o & 31));
        }
        __syncwarp();
      }
      clear_bitmap(sh.dirty, c + 1);
      __syncthreads();
      // B: completions -- for each propagating origin o', the items of column
      // o' waiting on a newly completed NT advance into this column
      bitmap_to_list(sh, sh.prop, c + 1);
      int np = sh.list_n;
      for (int i = warp; i < np; i += kWarps) {
        int o = sh.list[i];
        uint32_t* ex = sc.expn + (size_t)i * W;
        for (int w = lane; w < W; w += 32) ex[w] = 0;
        __syncwarp();
        for (int v = 0; v < VW; ++v) {
          uint32_t nw = sc.bnew[(size_t)o * VW + v];
          while (nw) {
            int b = __ffs(nw) - 1;
            nw &= nw - 1;
            int B = (v << 5) + b;
            for (int w = lane; w < W; w += 32) ex[w] |= g.exp_nt[(size_t)B * W + w];
          }
        }
        for (int v = lane; v < VW; v += 32) ws.bdone[(size_t)o * VW + v] |= sc.bnew[(size_t)o * VW + v];
        __syncwarp();
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        int s = 0;
        for (int i = 0; i < np; ++i) {
          int o = sh.list[i];
          sh.prefix[i] = s;
          s += ws.col_off[o + 1] - ws.col_off[o];
        }
        sh.prefix[np] = s;
      }
      __syncthreads();
      int total = sh.prefix[np];
      for (int t = warp; t < total; t += kWarps) {
        // find the propagating origin of pair t
        int lo = 0, hi = np - 1;
        while (lo < hi) {
          int mid = (lo + hi + 1) >> 1;
          if (sh.prefix[mid] <= t) lo = mid; else hi = mid - 1;
        }
        int o1 = sh.list[lo];
        int k = ws.col_off[o1] + (t - sh.prefix[lo]);
        int o = ws.org[k];
        bool nz = warp_scan_into(ws.stage + (size_t)o * W, ws.bits + (size_t)k * W,
                                 sc.expn + (size_t)lo * W, W, true, true);
        if (nz && lane == 0) {
          atomicOr(&sh.touched[o >> 5], 1u << (o & 31));
          atomicOr(&sh.next_dirty[o >> 5], 1u << (o & 31));
        }
      }
      clear_bitmap(sh.prop, c + 1);
      __syncthreads();
      // C: predictions for origin c from the nonterminals waited on here
      if (threadIdx.x == 0) {
        uint32_t any = 0;
        for (int v = 0; v < VW; ++v) any |= sh.vset[v] & ~sh.vdone[v];
        sh.changed = any != 0;
      }
      __syncthreads();
      if (sh.changed) {
        const uint32_t* P = gap ? g.gap_pred : g.pred;
        for (int w = threadIdx.x; w < W; w += blockDim.x) {
          uint32_t acc = 0;
          for (int v = 0; v < VW; ++v) {
            uint32_t nw = sh.vset[v] & ~sh.vdone[v];
            while (nw) {
              int b = __ffs(nw) - 1;
              nw &= nw - 1;
              acc |= P[(size_t)((v << 5) + b) * W + w];
            }
          }
          ws.stage[(size_t)c * W + w] |= acc;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
          for (int v = 0; v < VW; ++v) sh.vdone[v] |= sh.vset[v];
          sh.touched[c >> 5] |= 1u << (c & 31);
          sh.next_dirty[c >> 5] |= 1u << (c & 31);
        }
      }
      __syncthreads();
      for (int w = threadIdx.x; w < ((c + 32) >> 5); w += blockDim.x) {
        sh.dirty[w] = sh.next_dirty[w];
        sh.next_dirty[w] = 0;
      }
      __syncthreads();
    }
  }

  // Move the touched nonzero rows into the entry store as column c.
  __device__ void finish_column(int c) {
    int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    bitmap_to_list(sh, sh.touched, c + 1);
    int nl = sh.list_n;
    // nonzero flags into prefix
    for (int i = warp; i < nl; i += kWarps) {
      int o = sh.list[i];
      const uint32_t* row = ws.stage + (size_t)o * W;
      bool nz = false;
      for (int w = lane; w < W; w += 32) nz |= row[w] != 0;
      nz = __any_sync(0xffffffffu, nz);
      if (lane == 0) sh.prefix[i] = nz ? 1 : 0;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int s = 0;
      for (int i = 0; i < nl; ++i) {
        int f = sh.prefix[i];
        sh.prefix[i] = f ? s : -1;
        s += f;
      }
      long long base = ws.col_off[c];
      if (base + s > dims.emax) {
        sh.status = kWalkOverflow;
      } else {
        ws.col_off[c + 1] = (int)(base + s);
        sh.nent = base + s;
      }
      sh.ncols = c + 1;
    }
    __syncthreads();
    bool ok = sh.status != kWalkOverflow;
    int base = ws.col_off[c];
    for (int i = warp; i < nl; i += kWarps) {
      int o = sh.list[i];
      uint32_t* row = ws.stage + (size_t)o * W;
      int slot = sh.prefix[i];
      if (ok && slot >= 0) {
        if (lane == 0) ws.org[base + slot] = o;
        uint32_t* dst = ws.bits + (size_t)(base + slot) * W;
        for (int w = lane; w < W; w += 32) dst[w] = row[w];
        if constexpr (REC) record_entry(row, (long long)base + slot);
      }
      for (int w = lane; w < W; w += 32) row[w] = 0;
      for (int v = lane; v < VW; v += 32) ws.bdone[(size_t)o * VW + v] = 0;
    }
    clear_bitmap(sh.touched, c + 1);
    for (int v = threadIdx.x; v < VW; v += blockDim.x) {
      sh.vset[v] = 0;
      sh.vdone[v] = 0;
    }
    __syncthreads();
  }

  __device__ bool column_empty(int c) const { return ws.col_off[c + 1] == ws.col_off[c]; }

  // Warp: completed nonterminals and folded summaries of stored entry k.
  __device__ void record_entry(const uint32_t* row, long long k) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint32_t* nts = sh.wnt[warp];
    for (int v = lane; v < VW; v += 32) nts[v] = 0;
    __syncwarp();
    uint32_t fnt = 0, ft = 0;
    for (int w = lane; w < W; w += 32) {
      const uint32_t r = row[w];
      uint32_t m = r & g.complete[w];
      while (m) {
        const int b = __ffs(m) - 1;
        m &= m - 1;
        const int B = g.item_lhs[(w << 5) + b];
        atomicOr(&nts[B >> 5], 1u << (B & 31));
      }
      m = r & g.any_nt[w];
      while (m) {
        const int b = __ffs(m) - 1;
        m &= m - 1;
        fnt |= 1u << ((g.item_next[(w << 5) + b] - g.T) & 31);
      }
      m = r & g.any_term[w];
      while (m) {
        const int b = __ffs(m) - 1;
        m &= m - 1;
        ft |= 1u << (g.item_next[(w << 5) + b] & 31);
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
    int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    bitmap_to_list(sh, sh.touched, kMaxCols);
    int nl = sh.list_n;
    for (int i = warp; i < nl; i += kWarps) {
      int o = sh.list[i];
      for (int w = lane; w < W; w += 32) ws.stage[(size_t)o * W + w] = 0;
      for (int v = lane; v < VW; v += 32) ws.bdone[(size_t)o * VW + v] = 0;
    }
    clear_bitmap(sh.touched, kMaxCols);
    for (int v = threadIdx.x; v < VW; v += blockDim.x) {
      sh.vset[v] = 0;
      sh.vdone[v] = 0;
    }
    __syncthreads();
  }

  // Does column c hold the accept item with origin start_col?
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

using EarleyCols = EarleyColsT<false>;

}  // namespace epic

// Warp-level Earley walk: one warp recognizes one partial output.
//
// Same graph and chart as the block-wide walk (walk.cuh / skeleton.cuh), with
// every step done by one warp and no block barrier:
//  - a chart row is W words, lane l holding words l, l+32, ...;
//  - the closure of a column is a Gauss-Seidel sweep: completions from origin
//    o' only advance items of origins <= o', so the highest dirty origin is
//    closed first and its completions are pushed at once into lower rows;
//  - completed and waited-on nonterminals are read off a row with ballots;
//  - the span step groups lexings by (source, end state, terminals after the
//    first) chunk by chunk, lanes matching their keys against the groups made
//    so far.
#pragma once
#include "device.cuh"

namespace epic {

constexpr int kWarpsPerCta = 8;
constexpr int kWCols = 4096;    // columns per walk (graph nodes)
constexpr int kWMaxW = 256;
constexpr int kWMaxVW = 32;
constexpr int kWMaxQ = 1024;
constexpr long long kWMaxSteps = 1ll << 24;  // closure iterations per column

// index of (column j, origin o <= j) in a lower-triangular table
__host__ __device__ __forceinline__ size_t tri_index(int j, int o) { return (size_t)j * (j + 1) / 2 + o; }

struct WWs {  // per-warp global workspace
  uint32_t* stage;   // [nmax][W]
  uint32_t* bdone;   // [nmax][VW]
  int32_t* col_off;  // [nmax + 1]
  int32_t* org;      // [emax]
  uint32_t* esum;    // [emax][2] folded summaries of each entry (see row_scan)
  uint32_t* bits;    // [emax][W]
  uint32_t* ssum;    // [nmax][2] summaries of the stage rows (global staging)
  int32_t* f_q;      // [kWMaxQ]
  int32_t* f_c;      // [kWMaxQ]
  int32_t* g_src;    // [kWMaxQ]
  int32_t* g_end;    // [kWMaxQ]
  int32_t* g_len;    // [kWMaxQ]
  int32_t* g_last;   // [kWMaxQ]
  int32_t* key_q;    // [kWMaxQ]  representative of each end node (span step)
  uint32_t* g_tail;  // [kWMaxQ][4]  terminals 1..12 packed 4 per word
  uint32_t* g_lbl;   // [kWMaxQ][8]  first-terminal label set
};

// What a recording walk (a sequence's forward chart) writes besides the chart:
// the graph's edges in creation order of their target, gap flags, where each
// position's segment sits in the graph, and each entry's completed
// nonterminals.
struct SeqRec {
  uint8_t* col_gap;    // [nmax]
  int32_t* e_dst;      // [edge_cap]
  int32_t* e_src;      // [edge_cap]
  uint32_t* e_lbl;     // [edge_cap][8] terminal set of a labelled edge, all zero = epsilon
  int32_t* gap_col;    // [n] masked position -> column of its gap
  int32_t* pre_col;    // [n] fixed position -> column before its span (gap or BEGIN)
  int32_t* post_col;   // [n] fixed position -> column after its span (gap or END)
  uint32_t* cnt;       // [emax][VW] completed nonterminals of each entry
  int32_t* meta;       // [8]: ncols, nedges, start, accept, status, nent (low), -, -
  int edge_cap;
  int n_edges;         // running count (kept by the walk)
};

struct WSh {  // per-warp shared memory
  uint32_t touched[kWCols / 32];
  uint32_t dirty[kWCols / 32];
  uint32_t vset[kWMaxVW], vdone[kWMaxVW], nt[kWMaxVW];
  uint32_t vdone_tot[kWMaxVW];  // nonterminals newly completed from the origin being closed
  uint32_t lbl[kWMaxW];
  uint32_t expn[kWMaxW];
};

__device__ __forceinline__ uint32_t wl_lane() { return threadIdx.x & 31; }

// Warp: out[w] = items waiting on a member of the nonterminal set nts
// (VW words, readable by every lane), for the lane's words w.  A small set
// ORs its EXP_NT rows; a large one tests each item's next symbol instead
// (both give exactly the items whose next symbol is in the set).
__device__ __forceinline__ void expn_of_set(const DevGrammar& g, const uint32_t* nts, uint32_t* out) {
  const int W = g.W, VW = g.VW;
  int cnt = 0;
  for (int v = 0; v < VW; ++v) cnt += __popc(nts[v]);
  if (cnt <= 24) {
    for (int w = wl_lane(); w < W; w += 32) {
      uint32_t acc = 0;
      for (int v = 0; v < VW; ++v) {
        uint32_t m = nts[v];
        while (m) {
          const int b = __ffs(m) - 1;
          m &= m - 1;
          acc |= g.exp_nt[(size_t)((v << 5) + b) * W + w];
        }
      }
      out[w] = acc;
    }
  } else {
    for (int w = wl_lane(); w < W; w += 32) {
      uint32_t acc = 0;
      const int i0 = w << 5;
#pragma unroll 8
      for (int b = 0; b < 32; ++b) {
        const int i = i0 + b;
        const int s = i < g.D ? g.item_next[i] - g.T : -1;
        if (s >= 0 && ((nts[s >> 5] >> (s & 31)) & 1u)) acc |= 1u << b;
      }
      out[w] = acc;
    }
  }
}

#ifdef EPIC_PHASE_TIMERS
static __device__ unsigned long long g_phase[16];  // one per translation unit
#define PH_BEGIN(v) long long v = clock64()
#define PH_END(i, v)                                              \
  do {                                                            \
    if (wl_lane() == 0) atomicAdd(&g_phase[i], clock64() - (v)); \
  } while (0)
#else
#define PH_BEGIN(v)
#define PH_END(i, v)
#endif

// SM = true keeps the rows of the column under construction in shared memory
// (slot-mapped, rmax rows); SM = false keeps them in the per-warp global
// stage.  KWv item words per lane: rows of up to 32 KWv words.  EXT = true
// adds the base chart, the suffix mode and the recording of checks by region
// (compiled out of whole-graph walks).
template <bool SM, bool EXT = false, int KWv = (SM ? 1 : kWMaxW / 32)>
class WarpWalker {
  static constexpr int KW = KWv;  // item words per lane

 public:
  // shared-memory staging (SM): rows [rmax][W], completed-NT sets [rmax][VW],
  // slot of each origin (-1 = none) and origin of each slot
  uint32_t* srow = nullptr;
  uint32_t* sbdone = nullptr;
  int16_t* slot_of = nullptr;
  int32_t* slot_org = nullptr;
  uint32_t* slot_sum = nullptr;  // [rmax][2]
  int rmax = 0;
  int nslots = 0;
  const DevGrammar& g;
  const LexEntry* table;
  WWs ws;
  WSh& sh;
  int nmax;
  long long emax;
  int vocab;
  int W, VW;
  // walk state (uniform across the warp, kept in registers)
  int ncols;
  long long nent;
  int status;  // 0 ok, 1 overflow, 2 bad input
  int nf;
  int start_col;
  uint32_t label_fold = 0;  // bit (a mod 32) of every terminal in sh.lbl
  // A read-only base chart (a sequence's forward chart) holds columns
  // 0 .. base_cols-1 and entries 0 .. base_ent-1; this walk's own columns
  // follow with ids from base_cols.
  int base_cols = 0;
  long long base_ent = 0;
  const int32_t* b_col_off = nullptr;
  const int32_t* b_org = nullptr;
  const uint32_t* b_bits = nullptr;
  const uint32_t* b_esum = nullptr;
  // recording of the forward chart's graph (null when not recording)
  SeqRec* rec = nullptr;
  int cur_col = -1;
  uint32_t cur_lbl8[8];      // label set of the arrivals being made (all zero = epsilon)
  bool col_labelled = false; // the open column has a labelled arrival (else only epsilon ones)
  // Checks by region: the span step about to run is the region's last and
  // the node after it is a gap resolved by the base chart's good masks.  An
  // end node all of whose lexer states reach that gap by an epsilon edge is
  // then not closed: the gap's suffix-mode test (good masks include every
  // completion an item's closure makes, and the gap advances any waiting
  // item) gives the same answer for its rows as for their closure.
  bool defer_to_gap = false;
  // the pending lexeme at lexer state q reaches a following gap by an epsilon edge
  __device__ bool eps_into_gap(int q) const {
    const int a = g.dfa_accept[q];
    return q == 0 || g.dfa_ext[q] || (a >= 0 && g.skip[a]);
  }

  __device__ WarpWalker(const DevGrammar& g_, const LexEntry* t, WWs w, WSh& s, int nm, long long em, int voc)
      : g(g_), table(t), ws(w), sh(s), nmax(nm), emax(em), vocab(voc), W(g_.W), VW(g_.VW) {}

  __device__ void set_smem(uint32_t* rows, uint32_t* bd, int16_t* so, int32_t* sorg, uint32_t* ssum, int rm) {
    slot_sum = ssum;
    srow = rows;
    sbdone = bd;
    slot_of = so;
    slot_org = sorg;
    rmax = rm;
    for (int i = wl_lane(); i < nmax; i += 32) slot_of[i] = -1;
    nslots = 0;
    __syncwarp();
  }
  // stage row of origin o (allocating a zeroed slot for a new origin); null on overflow
  __device__ uint32_t* row_of(int o) {
    if constexpr (!SM) {
      return ws.stage + (size_t)o * W;
    } else {
      int sl = slot_of[o];
      if (sl < 0) {
        if (nslots >= rmax) {
          status = 1;
          return nullptr;
        }
        sl = nslots++;
        for (int w = wl_lane(); w < W; w += 32) srow[sl * W + w] = 0;
        for (int v = wl_lane(); v < VW; v += 32) sbdone[sl * VW + v] = 0;
        if (wl_lane() == 0) {
          slot_of[o] = (int16_t)sl;
          slot_org[sl] = o;
          slot_sum[sl * 2] = 0;
          slot_sum[sl * 2 + 1] = 0;
        }
        __syncwarp();
      }
      return srow + sl * W;
    }
  }
  // every slot of the open column goes back (also rows allocated but never
  // touched, whose origin would otherwise keep a stale slot)
  __device__ void release_slots() {
    if constexpr (SM) {
      for (int s2 = wl_lane(); s2 < nslots; s2 += 32) slot_of[slot_org[s2]] = -1;
      nslots = 0;
      __syncwarp();
    }
  }
  __device__ uint32_t* bdone_of(int o) {
    if constexpr (!SM) return ws.bdone + (size_t)o * VW;
    else return sbdone + slot_of[o] * VW;
  }
  __device__ uint32_t* sum_of(int o) {
    if constexpr (!SM) return ws.ssum + (size_t)o * 2;
    else return slot_sum + slot_of[o] * 2;
  }

  // ------------------------------------------------------------ chart access
  __device__ long long cbeg(int c) const {
    if constexpr (!EXT) return ws.col_off[c];
    return c < base_cols ? (long long)b_col_off[c] : base_ent + ws.col_off[c - base_cols];
  }
  __device__ long long cend(int c) const {
    if constexpr (!EXT) return ws.col_off[c + 1];
    return c < base_cols ? (long long)b_col_off[c + 1] : base_ent + ws.col_off[c - base_cols + 1];
  }
  __device__ int eorg(long long k) const {
    if constexpr (!EXT) return ws.org[k];
    return k < base_ent ? b_org[k] : ws.org[k - base_ent];
  }
  __device__ const uint32_t* ebits(long long k) const {
    if constexpr (!EXT) return ws.bits + (size_t)k * W;
    return k < base_ent ? b_bits + (size_t)k * W : ws.bits + (size_t)(k - base_ent) * W;
  }
  __device__ uint32_t esum(long long k, int which) const {
    if constexpr (!EXT) return ws.esum[(size_t)k * 2 + which];
    return k < base_ent ? b_esum[(size_t)k * 2 + which] : ws.esum[(size_t)(k - base_ent) * 2 + which];
  }

  // ------------------------------------------------------------ bitmaps
  __device__ void bm_clear(uint32_t* bm, int nbits) {
    for (int w = wl_lane(); w < ((nbits + 31) >> 5); w += 32) bm[w] = 0;
    __syncwarp();
  }
  __device__ void bm_set(uint32_t* bm, int i) {
    if (wl_lane() == 0) bm[i >> 5] |= 1u << (i & 31);
    __syncwarp();
  }
  // highest set bit below nbits, or -1
  __device__ int bm_highest(const uint32_t* bm, int nbits) {
    int nw = (nbits + 31) >> 5;
    for (int top = nw - 1; top >= 0; top -= 32) {
      int w = top - (int)wl_lane();
      uint32_t v = (w >= 0) ? bm[w] : 0u;
      unsigned any = __ballot_sync(0xffffffffu, v != 0);
      if (any) {
        int l = __ffs(any) - 1;  // lowest lane = highest word
        uint32_t vv = __shfl_sync(0xffffffffu, v, l);
        return ((top - l) << 5) + (31 - __clz(vv));
      }
    }
    return -1;
  }
  // lowest set bit at or above `from`, below nbits, or -1
  __device__ int bm_next(const uint32_t* bm, int from, int nbits) {
    int nw = (nbits + 31) >> 5;
    for (int base = from >> 5; base < nw; base += 32) {
      int w = base + (int)wl_lane();
      uint32_t v = (w < nw) ? bm[w] : 0u;
      if (w == (from >> 5)) v &= ~0u << (from & 31);
      unsigned any = __ballot_sync(0xffffffffu, v != 0);
      if (any) {
        int l = __ffs(any) - 1;
        uint32_t vv = __shfl_sync(0xffffffffu, v, l);
        return ((base + l) << 5) + (__ffs(vv) - 1);
      }
    }
    return -1;
  }

  // ------------------------------------------------------------ row ops
  // row |= shift(row & M), until stable (item (p, d) -> (p, d+1)); the row is
  // held in registers (lane l owns words l, l+32, ...) while it is iterated
  __device__ void row_advance(uint32_t* row, const uint32_t* M) {
    const int nw = (W + 31) >> 5;
    const int lane = wl_lane();
    uint32_t r[KW], m[KW];
#pragma unroll
    for (int i = 0; i < KW; ++i) {
      int w = lane + 32 * i;
      bool ok = i < nw && w < W;
      r[i] = ok ? row[w] : 0u;
      m[i] = ok ? M[w] : 0u;
    }
    bool any_change = false;
    for (int it = 0; it < 64; ++it) {
      bool ch = false;
      uint32_t carry = 0;
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        if (i < nw) {
          uint32_t v = r[i] & m[i];
          uint32_t prev = __shfl_up_sync(0xffffffffu, v, 1);
          if (lane == 0) prev = carry;
          carry = __shfl_sync(0xffffffffu, v, 31);
          uint32_t add = ((v << 1) | (prev >> 31)) & ~r[i];
          ch |= add != 0;
          r[i] |= add;
        }
      }
      if (!__any_sync(0xffffffffu, ch)) break;
      any_change = true;
    }
    if (any_change) {
#pragma unroll
      for (int i = 0; i < KW; ++i) {
        int w = lane + 32 * i;
        if (i < nw && w < W) row[w] = r[i];
      }
    }
    __syncwarp();
  }
  // dst |= shift(src & M) (or src & M / src); marks origin o; returns nonzero
  __device__ bool row_into(uint32_t* dst, const uint32_t* src, const uint32_t* M, bool shift) {
    bool nz = false;
    uint32_t carry = 0;
    for (int base = 0; base < W; base += 32) {
      int w = base + wl_lane();
      uint32_t v = (w < W) ? (M ? (src[w] & M[w]) : src[w]) : 0u;
      uint32_t add = v;
      if (shift) {
        uint32_t prev = __shfl_up_sync(0xffffffffu, v, 1);
        if (wl_lane() == 0) prev = carry;
        add = (v << 1) | (prev >> 31);
        carry = __shfl_sync(0xffffffffu, v, 31);
      }
      if (w < W && add) {
        uint32_t old = dst[w];
        if ((old | add) != old) {
          dst[w] = old | add;
          nz = true;
        }
      }
    }
    __syncwarp();
    return __any_sync(0xffffffffu, nz);
  }
  // nonterminal set of the items of `row` selected by mask (via lhs or next
  // symbol), ORed into out (VW words in shared memory)
  __device__ void row_nts(const uint32_t* row, const uint32_t* mask, bool by_lhs, uint32_t* out) {
    for (int base = 0; base < W; base += 32) {
      int w = base + wl_lane();
      uint32_t m = (w < W) ? (row[w] & mask[w]) : 0u;
      unsigned nzl = __ballot_sync(0xffffffffu, m != 0);
      while (nzl) {
        int s = __ffs(nzl) - 1;
        nzl &= nzl - 1;
        uint32_t mm = __shfl_sync(0xffffffffu, m, s);
        if ((mm >> wl_lane()) & 1u) {
          int item = ((base + s) << 5) + wl_lane();
          int B = by_lhs ? g.item_lhs[item] : (g.item_next[item] - g.T);
          atomicOr(&out[B >> 5], 1u << (B & 31));
        }
      }
    }
    __syncwarp();
  }

  // One pass over a row: the nonterminals its items wait on (ORed into the
  // exact set `vs`) and two folded 32-bit summaries -- bit (B mod 32) for a
  // waited-on nonterminal B, bit (a mod 32) for an expected terminal a --
  // used to skip chart entries that cannot take part in a completion or a
  // scan (a superset filter, exact for up to 32 symbols).
  __device__ void row_scan(const uint32_t* row, uint32_t* vs, uint32_t* sum2) {
    uint32_t fnt = 0, ft = 0;
    for (int base = 0; base < W; base += 32) {
      int w = base + wl_lane();
      uint32_t r = (w < W) ? row[w] : 0u;
      uint32_t mn = (w < W) ? (r & g.any_nt[w]) : 0u;
      uint32_t mt = (w < W) ? (r & g.any_term[w]) : 0u;
      unsigned nzl = __ballot_sync(0xffffffffu, (mn | mt) != 0);
      while (nzl) {
        int s = __ffs(nzl) - 1;
        nzl &= nzl - 1;
        uint32_t a = __shfl_sync(0xffffffffu, mn, s);
        uint32_t b = __shfl_sync(0xffffffffu, mt, s);
        int item = ((base + s) << 5) + wl_lane();
        if ((a >> wl_lane()) & 1u) {
          int B = g.item_next[item] - g.T;
          atomicOr(&vs[B >> 5], 1u << (B & 31));
          fnt |= 1u << (B & 31);
        }
        if ((b >> wl_lane()) & 1u) ft |= 1u << (g.item_next[item] & 31);
      }
    }
    for (int off = 16; off; off >>= 1) {
      fnt |= __shfl_xor_sync(0xffffffffu, fnt, off);
      ft |= __shfl_xor_sync(0xffffffffu, ft, off);
    }
    if (wl_lane() == 0) {
      sum2[0] = fnt;
      sum2[1] = ft;
    }
    __syncwarp();
  }

  // Scatter the entries of finished column `col` into the stage, one entry per
  // lane: dst(org) |= shift(bits & M) (or bits & M, or bits).  Entries of one
  // column have distinct origins, so lanes never share a destination row.
  // `which` selects the summary filter (0: waited nonterminals, 1: expected
  // terminals, -1: none) tested against `fold`.
  __device__ void scatter(int col, const uint32_t* M, bool shift, int which, uint32_t fold, int skip_org = -1) {
    const int lane = wl_lane();
    const long long b = cbeg(col), e = skip_org >= 0 ? cend(col) - 1 : cend(col);
    if (!SM && W > 16) {  // wide rows in the global stage: the lanes share each entry's words
      for (long long base = b; base < e; base += 32) {
        const long long k = base + lane;
        const bool act = k < e && (which < 0 || (esum(k, which) & fold) != 0);
        unsigned am = __ballot_sync(0xffffffffu, act);
        const int my_org = act ? eorg(k) : -1;
        while (am) {  // up to four entries at a time: their loads overlap
          int ls[4];
          int nl = 0;
          while (am && nl < 4) {
            ls[nl++] = __ffs(am) - 1;
            am &= am - 1;
          }
          const uint32_t* src[4];
          uint32_t* dst[4];
          int o2[4];
          uint32_t carry[4];
          bool ch[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int l = i < nl ? ls[i] : ls[0];
            o2[i] = __shfl_sync(0xffffffffu, my_org, l);
            src[i] = ebits(base + l);
            dst[i] = i < nl ? row_of(o2[i]) : nullptr;
            carry[i] = 0;
            ch[i] = false;
          }
          if (status) return;  // no shared-memory slot left
          for (int w0 = 0; w0 < W; w0 += 32) {
            const int w = w0 + lane;
            const uint32_t m = (M && w < W) ? M[w] : 0xffffffffu;
            uint32_t v[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) v[i] = (i < nl && w < W) ? (src[i][w] & m) : 0u;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              uint32_t add = v[i];
              if (shift) {
                uint32_t prev = __shfl_up_sync(0xffffffffu, v[i], 1);
                if (lane == 0) prev = carry[i];
                add = (v[i] << 1) | (prev >> 31);
                carry[i] = __shfl_sync(0xffffffffu, v[i], 31);
              }
              if (i < nl && w < W && add) {
                const uint32_t old = dst[i][w];
                if ((old | add) != old) {
                  dst[i][w] = old | add;
                  ch[i] = true;
                }
              }
            }
          }
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const bool any = __any_sync(0xffffffffu, ch[i]);
            if (i < nl && any && lane == 0) {
              sh.touched[o2[i] >> 5] |= 1u << (o2[i] & 31);
              sh.dirty[o2[i] >> 5] |= 1u << (o2[i] & 31);
            }
          }
          __syncwarp();
        }
      }
      return;
    }
    for (long long base = b; base < e; base += 32) {
      long long k = base + lane;
      bool act = k < e && (which < 0 || (esum(k, which) & fold) != 0);
      unsigned am = __ballot_sync(0xffffffffu, act);
      if (!am) continue;
      int o2 = act ? eorg(k) : -1;
      uint32_t* dst = nullptr;
      if constexpr (SM) {
        bool need = act && slot_of[o2] < 0;
        unsigned nm = __ballot_sync(0xffffffffu, need);
        int nneed = __popc(nm);
        if (nslots + nneed > rmax) {
          status = 1;
          return;
        }
        if (need) {
          int sl = nslots + __popc(nm & ((1u << lane) - 1u));
          slot_of[o2] = (int16_t)sl;
          slot_org[sl] = o2;
          slot_sum[sl * 2] = 0;
          slot_sum[sl * 2 + 1] = 0;
          for (int w = 0; w < W; ++w) srow[sl * W + w] = 0;
          for (int v = 0; v < VW; ++v) sbdone[sl * VW + v] = 0;
        }
        nslots += nneed;
        __syncwarp();
        if (act) dst = srow + slot_of[o2] * W;
      } else {
        if (act) dst = ws.stage + (size_t)o2 * W;
      }
      bool ch = false;
      if (act) {
        const uint32_t* src = ebits(k);
        uint32_t carry = 0;
        for (int w = 0; w < W; ++w) {
          uint32_t v = M ? (src[w] & M[w]) : src[w];
          uint32_t add = shift ? ((v << 1) | carry) : v;
          carry = v >> 31;
          if (add) {
            uint32_t old = dst[w];
            if ((old | add) != old) {
              dst[w] = old | add;
              ch = true;
            }
          }
        }
        if (ch) {
          atomicOr(&sh.touched[o2 >> 5], 1u << (o2 & 31));
          atomicOr(&sh.dirty[o2 >> 5], 1u << (o2 & 31));
        }
      }
      __syncwarp();
    }
  }

  // row |= shift(items of E waiting on a member of the nonterminal set nts);
  // returns whether row changed
  __device__ bool row_into_waiting(uint32_t* row, const uint32_t* E, const uint32_t* nts) {
    bool ch = false;
    uint32_t carry = 0;
    for (int base = 0; base < W; base += 32) {
      const int w = base + wl_lane();
      uint32_t x = 0;
      if (w < W) {
        uint32_t m = E[w] & g.any_nt[w];
        while (m) {
          const int b = __ffs(m) - 1;
          m &= m - 1;
          const int B = g.item_next[(w << 5) + b] - g.T;
          if ((nts[B >> 5] >> (B & 31)) & 1u) x |= 1u << b;
        }
      }
      uint32_t prev = __shfl_up_sync(0xffffffffu, x, 1);
      if (wl_lane() == 0) prev = carry;
      carry = __shfl_sync(0xffffffffu, x, 31);
      const uint32_t add = (x << 1) | (prev >> 31);
      if (w < W && add) {
        const uint32_t old = row[w];
        if ((old | add) != old) {
          row[w] = old | add;
          ch = true;
        }
      }
    }
    __syncwarp();
    return __any_sync(0xffffffffu, ch);
  }

  // ------------------------------------------------------------ columns
  __device__ int open_column() {
    if (ncols >= nmax) {
      status = 1;
      return -1;
    }
    cur_col = ncols;
    return ncols;
  }
  __device__ void arrive(int src, const uint32_t* M, bool shift) {
    PH_BEGIN(t_arr);
    arrive_inner(src, M, shift);
    PH_END(1, t_arr);
  }
  __device__ void record_edge(int src, bool labelled) {
    if (wl_lane() == 0) {
      if (rec->n_edges >= rec->edge_cap) {
        status = 1;
      } else {
        int e = rec->n_edges++;
        rec->e_dst[e] = cur_col;
        rec->e_src[e] = src;
        for (int w = 0; w < 8; ++w) rec->e_lbl[(size_t)e * 8 + w] = labelled ? cur_lbl8[w] : 0u;
      }
    }
    status = __shfl_sync(0xffffffffu, status, 0);
    rec->n_edges = __shfl_sync(0xffffffffu, rec->n_edges, 0);
  }
  __device__ void arrive_inner(int src, const uint32_t* M, bool shift) {
    col_labelled |= shift;
    if constexpr (EXT)
      if (rec) record_edge(src, shift);
    if (shift)
      scatter(src, M, true, 1, label_fold);
    else
      scatter(src, M, false, -1, 0u);
  }
  __device__ void seed(int c) {
    uint32_t* r = row_of(c);
    if (!r) return;
    if (wl_lane() == 0) r[g.start_item >> 5] |= 1u << (g.start_item & 31);
    __syncwarp();
    bm_set(sh.touched, c);
    bm_set(sh.dirty, c);
  }

  // Suffix mode (a check's nodes after its region): no predictions, and rows
  // whose origin is a base-chart column are not closed here -- whether such
  // an item leads to acceptance is read from the base chart's good masks at
  // node res_node when the column is finished (found = 1); they are not kept.
  bool suffix_mode = false;
  int res_node = -1;
  const uint32_t* good = nullptr;
  int found = 0;
  int region_start = -1;  // own start column (S' item has an own origin) or -1
  int accept_node = -1;   // the base chart's accept node

  // entry of base-chart column j with origin o, or -1
  const int32_t* b_eidx = nullptr;  // [(j (j + 1) / 2) + o] for o <= j
  __device__ long long find_base(int j, int o) const { return o > j ? -1 : (long long)b_eidx[tri_index(j, o)]; }

  bool cur_gap = false;
  __device__ void close_column(int c, bool gap) {
    cur_gap = gap;
    const uint32_t* P = gap ? g.gap_pred : g.pred;
    // A node (not a gap) reached only by epsilon edges from finished columns:
    // each row below c is a union of rows closed under completion and
    // advance, and so is the union, so those rows only contribute their
    // waited nonterminals (the predictions at c).
    const bool eps_only = !gap && !col_labelled;
    for (long long it = 0;; ++it) {
      if (it > kWMaxSteps) {
        status = 1;
        return;
      }
      int o = bm_highest(sh.dirty, c + 1);
      if (EXT && suffix_mode) {
        if (o < 0) break;
        if (o < base_cols) {  // resolved by the good masks at finish
          if (wl_lane() == 0) sh.dirty[o >> 5] &= ~(1u << (o & 31));
          __syncwarp();
          continue;
        }
      }
      if (o < 0) {
        // predictions for origin c from the nonterminals waited on here
        bool any = false;
        for (int v = wl_lane(); v < VW; v += 32) any |= (sh.vset[v] & ~sh.vdone[v]) != 0;
        if (!__any_sync(0xffffffffu, any)) break;
        uint32_t* crow = row_of(c);
        if (!crow) return;
        for (int w = wl_lane(); w < W; w += 32) {
          uint32_t acc = 0;
          for (int v = 0; v < VW; ++v) {
            uint32_t nw = sh.vset[v] & ~sh.vdone[v];
            while (nw) {
              int b = __ffs(nw) - 1;
              nw &= nw - 1;
              acc |= P[(size_t)((v << 5) + b) * W + w];
            }
          }
          crow[w] |= acc;
        }
        __syncwarp();
        for (int v = wl_lane(); v < VW; v += 32) sh.vdone[v] |= sh.vset[v];
        __syncwarp();
        bm_set(sh.touched, c);
        bm_set(sh.dirty, c);
        continue;
      }
      if (wl_lane() == 0) sh.dirty[o >> 5] &= ~(1u << (o & 31));
      __syncwarp();
      uint32_t* row = row_of(o);
      if (eps_only && o < c) {
        row_scan(row, sh.vset, sum_of(o));
        continue;
      }
      if (o == c) {  // completions from c at c: the nullable / gap advance rules
        PH_BEGIN(t_row);
        row_advance(row, gap ? g.next_any : g.nullable_next);
        PH_END(3, t_row);
        row_scan(row, sh.vset, sum_of(o));
        continue;
      }
      // Completions from o advance the items of column o; of those, only the
      // entry with origin o itself (the last one: entries are stored by
      // ascending origin) feeds row o again.  Close that loop first, then
      // scatter everything completed from o once over the other entries.
      const long long ke = cend(o);
      const bool self = ke > cbeg(o) && eorg(ke - 1) == o;
      uint32_t* bd = bdone_of(o);
      for (int v = wl_lane(); v < VW; v += 32) sh.vdone_tot[v] = 0;
      bool any_tot = false;
      for (int round = 0; round < 64 * kWMaxW; ++round) {
        PH_BEGIN(t_row);
        row_advance(row, gap ? g.next_any : g.nullable_next);
        PH_END(3, t_row);
        PH_BEGIN(t_nts);
        for (int v = wl_lane(); v < VW; v += 32) sh.nt[v] = 0;
        __syncwarp();
        row_nts(row, g.complete, true, sh.nt);
        bool any = false;
        for (int v = wl_lane(); v < VW; v += 32) {
          const uint32_t d = sh.nt[v] & ~bd[v];
          sh.nt[v] = d;
          any |= d != 0;
          bd[v] |= d;
          sh.vdone_tot[v] |= d;
        }
        __syncwarp();
        PH_END(4, t_nts);
        any = __any_sync(0xffffffffu, any);
        any_tot |= any;
        if (!any || !self) break;
        if (!row_into_waiting(row, ebits(ke - 1), sh.nt)) break;
      }
      row_scan(row, sh.vset, sum_of(o));
      if (!any_tot) continue;
      PH_BEGIN(t_expn);
      // EXPN: items waiting on a nonterminal newly completed from o
      expn_of_set(g, sh.vdone_tot, sh.expn);
      __syncwarp();
      PH_END(5, t_expn);
      PH_BEGIN(t_part);
      uint32_t fold = 0;
      for (int v = 0; v < VW; ++v) fold |= sh.vdone_tot[v];
      scatter(o, sh.expn, true, 0, fold, self ? o : -1);
      if (status) return;
      PH_END(6, t_part);
    }
  }

  __device__ void finish_column(int c) {
    PH_BEGIN(t_fin);
    finish_inner(c);
    PH_END(7, t_fin);
  }
  __device__ void finish_inner(int c) {
    const int oc = c - base_cols;  // own column index
    long long E = ws.col_off[oc];
    int o = -1;
    while ((o = bm_next(sh.touched, o + 1, c + 1)) >= 0) {
      uint32_t* row = row_of(o);
      bool nz = false;
      for (int w = wl_lane(); w < W; w += 32) nz |= row[w] != 0;
      nz = __any_sync(0xffffffffu, nz);
      if (EXT && nz && suffix_mode && o < base_cols) {
        long long kf = find_base(res_node, o);
        bool hit = false;
        if (kf >= 0)
          for (int w = wl_lane(); w < W; w += 32) hit |= (row[w] & good[(size_t)kf * W + w]) != 0;
        if (__any_sync(0xffffffffu, hit)) found = 1;
        nz = false;  // not kept
      }
      if (EXT && nz && suffix_mode && o == region_start && res_node == accept_node &&
          ((row[g.accept_item >> 5] >> (g.accept_item & 31)) & 1u))
        found = 1;
      if (nz) {
        if (E >= emax) {
          status = 1;
        } else {
          if (wl_lane() == 0) {
            ws.org[E] = o;
            uint32_t* sm = sum_of(o);
            ws.esum[(size_t)E * 2] = sm[0];
            ws.esum[(size_t)E * 2 + 1] = sm[1];
          }
          uint32_t* dst = ws.bits + (size_t)E * W;
          for (int w = wl_lane(); w < W; w += 32) dst[w] = row[w];
          if (EXT && rec) {  // completed nonterminals of the entry
            for (int v = wl_lane(); v < VW; v += 32) sh.nt[v] = 0;
            __syncwarp();
            row_nts(row, g.complete, true, sh.nt);
            for (int v = wl_lane(); v < VW; v += 32) rec->cnt[(size_t)E * VW + v] = sh.nt[v];
          }
          ++E;
        }
      }
      if constexpr (!SM) {
        for (int w = wl_lane(); w < W; w += 32) row[w] = 0;
        for (int v = wl_lane(); v < VW; v += 32) ws.bdone[(size_t)o * VW + v] = 0;
      }
    }
    release_slots();
    bm_clear(sh.touched, c + 1);
    for (int v = wl_lane(); v < VW; v += 32) {
      sh.vset[v] = 0;
      sh.vdone[v] = 0;
    }
    if (wl_lane() == 0) {
      ws.col_off[oc + 1] = (int)E;
      if (EXT && rec) rec->col_gap[c] = cur_gap ? 1 : 0;
    }
    __syncwarp();
    nent = E;
    ncols = c + 1;
    col_labelled = false;
  }
  __device__ bool column_empty(int c) { return cend(c) == cbeg(c); }

  // abandon the open column: zero its rows
  __device__ void cleanup() {
    col_labelled = false;
    int o = -1;
    while ((o = bm_next(sh.touched, o + 1, kWCols)) >= 0) {
      if constexpr (!SM) {
        for (int w = wl_lane(); w < W; w += 32) ws.stage[(size_t)o * W + w] = 0;
        for (int v = wl_lane(); v < VW; v += 32) ws.bdone[(size_t)o * VW + v] = 0;
      }
    }
    release_slots();
    bm_clear(sh.touched, kWCols);
    bm_clear(sh.dirty, kWCols);
    for (int v = wl_lane(); v < VW; v += 32) {
      sh.vset[v] = 0;
      sh.vdone[v] = 0;
    }
    __syncwarp();
  }

  __device__ bool accepts(int c, int start) {
    bool f = false;
    for (long long k = cbeg(c) + wl_lane(); k < cend(c); k += 32)
      if (eorg(k) == start && ((ebits(k)[g.accept_item >> 5] >> (g.accept_item & 31)) & 1u)) f = true;
    return __any_sync(0xffffffffu, f);
  }

  // ------------------------------------------------------------ labels
  __device__ void label_set(const uint32_t* lbl8) {
    label_fold = 0;
    for (int lw = 0; lw < 8; ++lw) {
      label_fold |= lbl8[lw];
      cur_lbl8[lw] = lbl8[lw];
    }
    for (int w = wl_lane(); w < W; w += 32) {
      uint32_t acc = 0;
      for (int lw = 0; lw < 8; ++lw) {
        uint32_t m = lbl8[lw];
        while (m) {
          int b = __ffs(m) - 1;
          m &= m - 1;
          int a = (lw << 5) + b;
          if (a < g.T) acc |= g.exp_term[(size_t)a * W + w];
        }
      }
      sh.lbl[w] = acc;
    }
    __syncwarp();
  }
  __device__ void label_one(int a) {
    label_fold = 1u << (a & 31);
    for (int lw = 0; lw < 8; ++lw) cur_lbl8[lw] = (lw == (a >> 5)) ? (1u << (a & 31)) : 0u;
    for (int w = wl_lane(); w < W; w += 32) sh.lbl[w] = g.exp_term[(size_t)a * W + w];
    __syncwarp();
  }

  // a node built from labelled / epsilon arrivals, closed and stored
  __device__ bool simple_column(int& c_out, int src, bool eps, bool gap) {
    int c = open_column();
    if (c < 0) return false;
    arrive(src, eps ? nullptr : sh.lbl, !eps);
    close_column(c, gap);
    finish_column(c);
    c_out = c;
    return status == 0;
  }

  // ------------------------------------------------------------ span step
  __device__ static uint32_t tail_word(const LexEntry& e, int i) {
    uint32_t v = 0;
    for (int j = 0; j < 4; ++j) {
      int t = 1 + 4 * i + j;
      v |= (uint32_t)(t < e.len ? e.term[t] : 0) << (8 * j);
    }
    return v;
  }

  __device__ bool span_step(int tok) {
    if (g.lazy.stats && wl_lane() == 0) atomicAdd(&g.lazy.stats[0], (unsigned long long)nf);
    int ng = 0;
    PH_BEGIN(t_group);
    // grouping, 32 frontier elements at a time
    for (int base = 0; base < nf; base += 32) {
      int f = base + (int)wl_lane();
      bool live = false;
      LexEntry e;
      int src = -1;
      if (f < nf) {
        e = lex_at(g, table, tok, ws.f_q[f]);
        src = ws.f_c[f];
        live = e.end != 0xFFFF;
      }
      uint32_t t0 = live ? tail_word(e, 0) : 0, t1 = live ? tail_word(e, 1) : 0, t2 = live ? tail_word(e, 2) : 0;
      int gid = -1;
      if (live) {
        for (int gi = 0; gi < ng; ++gi) {
          if (ws.g_src[gi] == src && ws.g_end[gi] == e.end && ws.g_len[gi] == e.len &&
              ws.g_tail[gi * 4] == t0 && ws.g_tail[gi * 4 + 1] == t1 && ws.g_tail[gi * 4 + 2] == t2) {
            gid = gi;
            break;
          }
        }
      }
      unsigned pending = __ballot_sync(0xffffffffu, live && gid < 0);
      while (pending) {
        int l = __ffs(pending) - 1;
        int ksrc = __shfl_sync(0xffffffffu, src, l);
        int kend = __shfl_sync(0xffffffffu, (int)(live ? e.end : 0), l);
        int klen = __shfl_sync(0xffffffffu, (int)(live ? e.len : 0), l);
        uint32_t k0 = __shfl_sync(0xffffffffu, t0, l), k1 = __shfl_sync(0xffffffffu, t1, l),
                 k2 = __shfl_sync(0xffffffffu, t2, l);
        if (ng >= kWMaxQ) {
          status = 1;
          return false;
        }
        if (wl_lane() == 0) {
          ws.g_src[ng] = ksrc;
          ws.g_end[ng] = kend;
          ws.g_len[ng] = klen;
          ws.g_tail[ng * 4] = k0;
          ws.g_tail[ng * 4 + 1] = k1;
          ws.g_tail[ng * 4 + 2] = k2;
          for (int w = 0; w < 8; ++w) ws.g_lbl[ng * 8 + w] = 0;
        }
        __syncwarp();
        bool same = live && gid < 0 && src == ksrc && (int)e.end == kend && (int)e.len == klen && t0 == k0 &&
                    t1 == k1 && t2 == k2;
        if (same) gid = ng;
        pending &= ~__ballot_sync(0xffffffffu, same);
        ++ng;
      }
      if (live && e.len > 0) atomicOr(&ws.g_lbl[gid * 8 + (e.term[0] >> 5)], 1u << (e.term[0] & 31));
      __syncwarp();
    }
    PH_END(0, t_group);
    // intermediate nodes: the run up to its last terminal; groups with the
    // same source, first-terminal set and terminals before the last one
    // spell the same paths up to it, so they share one chain of nodes
    for (int gi = 0; gi < ng; ++gi) {
      int len = ws.g_len[gi];
      int cur = ws.g_src[gi];
      if (len >= 2) {
        int share = -1;
        for (int gb = 0; gb < gi && share < 0; gb += 32) {
          const int gj = gb + (int)wl_lane();
          bool same = gj < gi && ws.g_len[gj] == len && ws.g_src[gj] == cur;
          for (int w = 0; w < 8 && same; ++w) same = ws.g_lbl[gj * 8 + w] == ws.g_lbl[gi * 8 + w];
          for (int t = 1; t + 1 < len && same; ++t) same = tail_term(gj, t) == tail_term(gi, t);
          const unsigned m = __ballot_sync(0xffffffffu, same);
          if (m) share = gb + __ffs(m) - 1;
        }
        if (share >= 0) {
          if (wl_lane() == 0) ws.g_last[gi] = ws.g_last[share];
          __syncwarp();
          continue;
        }
      }
      for (int t = 0; t + 1 < len; ++t) {
        if (t == 0) {
          label_set(ws.g_lbl + gi * 8);
        } else {
          uint32_t tw = ws.g_tail[gi * 4 + ((t - 1) >> 2)];
          label_one((tw >> (8 * ((t - 1) & 3))) & 0xff);
        }
        int c;
        if (!simple_column(c, cur, false, false)) return false;
        cur = c;
      }
      if (wl_lane() == 0) ws.g_last[gi] = cur;
      __syncwarp();
    }
    // the distinct end states, ascending (the old frontier is consumed)
    int nt = 0;
    int prev = -1;
    for (;;) {
      int best = 0x7fffffff;
      for (int gi = wl_lane(); gi < ng; gi += 32) {
        int e = ws.g_end[gi];
        if (e > prev && e < best) best = e;
      }
      for (int off = 16; off; off >>= 1) best = min(best, __shfl_xor_sync(0xffffffffu, best, off));
      if (best == 0x7fffffff) break;
      if (wl_lane() == 0) ws.f_q[nt] = best;
      ++nt;
      prev = best;
    }
    __syncwarp();
    // end nodes with the same arrivals (sources and labels) have the same
    // incoming paths: one column serves all their lexer states; the smallest
    // equal end is the representative (ws.f_c holds a hash of the arrivals
    // until the columns are made)
    for (int ti = wl_lane(); ti < nt; ti += 32) ws.f_c[ti] = (int32_t)arrivals_hash(ws.f_q[ti], ng);
    __syncwarp();
    for (int ti = wl_lane(); ti < nt; ti += 32) {
      int rep = ti;
      for (int tj = 0; tj < ti; ++tj)
        if (ws.f_c[tj] == ws.f_c[ti] && same_arrivals(ws.f_q[ti], ws.f_q[tj], ng)) {
          rep = tj;
          break;
        }
      ws.key_q[ti] = rep;
    }
    __syncwarp();
    for (int ti = 0; ti < nt; ++ti) {
      if (ws.key_q[ti] != ti) continue;
      const int best = ws.f_q[ti];
      int c = open_column();
      if (c < 0) return false;
      for (int gi = 0; gi < ng; ++gi) {
        if (ws.g_end[gi] != best) continue;
        int len = ws.g_len[gi];
        if (len == 0) {
          arrive(ws.g_src[gi], nullptr, false);
        } else if (len == 1) {
          label_set(ws.g_lbl + gi * 8);
          arrive(ws.g_src[gi], sh.lbl, true);
        } else {
          label_one(tail_term(gi, len - 1));
          arrive(ws.g_last[gi], sh.lbl, true);
        }
      }
      bool defer = false;
      if (EXT && defer_to_gap) {
        bool all_eps = true;
        for (int tj = (int)wl_lane(); tj < nt; tj += 32)
          if (ws.key_q[tj] == ti && !eps_into_gap(ws.f_q[tj])) all_eps = false;
        defer = __all_sync(0xffffffffu, all_eps);
      }
      if (defer) {
        // rows as they arrived: only their summaries (scatter filters)
        int o = -1;
        while ((o = bm_next(sh.touched, o + 1, c + 1)) >= 0) row_scan(row_of(o), sh.vset, sum_of(o));
        bm_clear(sh.dirty, c + 1);
      } else {
        close_column(c, false);
      }
      finish_column(c);
      if (status) return false;
      if (wl_lane() == 0) ws.f_c[ti] = c;
      __syncwarp();
    }
    // the new frontier: (end state, column) of the non-empty columns
    for (int ti = wl_lane(); ti < nt; ti += 32)
      if (ws.key_q[ti] != ti) ws.f_c[ti] = ws.f_c[ws.key_q[ti]];  // representatives are columns by now
    __syncwarp();
    int nk = 0;
    for (int ti = 0; ti < nt; ++ti) {
      const int c = ws.f_c[ti];
      if (column_empty(c)) continue;
      if (wl_lane() == 0) {
        ws.f_q[nk] = ws.f_q[ti];
        ws.f_c[nk] = c;
      }
      __syncwarp();
      ++nk;
    }
    nf = nk;
    return true;
  }

  // terminal t (1 .. len-1) of group gi's run
  __device__ int tail_term(int gi, int t) const {
    return (ws.g_tail[gi * 4 + ((t - 1) >> 2)] >> (8 * ((t - 1) & 3))) & 0xff;
  }
  // arrival of group gi into its end node: source column and label set (all
  // zero: epsilon)
  __device__ int arrival_src(int gi) const { return ws.g_len[gi] >= 2 ? ws.g_last[gi] : ws.g_src[gi]; }
  __device__ uint32_t arrival_lbl(int gi, int w) const {
    const int len = ws.g_len[gi];
    if (len == 0) return 0u;
    if (len == 1) return ws.g_lbl[gi * 8 + w];
    const int a = tail_term(gi, len - 1);
    return (w == (a >> 5)) ? (1u << (a & 31)) : 0u;
  }
  __device__ uint32_t arrivals_hash(int e, int ng) const {
    uint32_t h = 0;
    for (int gi = 0; gi < ng; ++gi) {
      if (ws.g_end[gi] != e) continue;
      uint32_t x = (uint32_t)arrival_src(gi) * 0x9E3779B1u + (ws.g_len[gi] == 0 ? 0x85EBCA6Bu : 0u);
      for (int w = 0; w < 8; ++w) x = (x ^ arrival_lbl(gi, w)) * 0xC2B2AE35u + (uint32_t)w;
      h += x ^ (x >> 16);
    }
    return h;
  }
  // do end states e1 and e2 receive the same arrivals?  (one lane)
  __device__ bool same_arrivals(int e1, int e2, int ng) const {
    int n1 = 0, n2 = 0;
    for (int gi = 0; gi < ng; ++gi) {
      n1 += ws.g_end[gi] == e1;
      n2 += ws.g_end[gi] == e2;
    }
    if (n1 != n2) return false;
    for (int gi = 0; gi < ng; ++gi) {
      if (ws.g_end[gi] != e1) continue;
      bool found = false;
      for (int gj = 0; gj < ng && !found; ++gj) {
        if (ws.g_end[gj] != e2 || arrival_src(gj) != arrival_src(gi)) continue;
        bool same = (ws.g_len[gi] == 0) == (ws.g_len[gj] == 0);
        for (int w = 0; w < 8; ++w) same &= arrival_lbl(gi, w) == arrival_lbl(gj, w);
        found = same;
      }
      if (!found) return false;
    }
    return true;
  }

  // ------------------------------------------------------------ the walk
  __device__ static int token_at(const int32_t* x, int sp, int st, int i) { return i == sp ? st : x[i]; }

  // x (+) {(sp, st)}; returns 1 valid, 0 invalid, -1 overflow, -2 bad input
  __device__ int run(const int32_t* x, int n, int sp, int st) {
    ncols = base_cols;
    nent = 0;
    status = 0;
    nf = 0;
    if (wl_lane() == 0) ws.col_off[0] = 0;
    __syncwarp();
    if (sp >= 0 && (sp >= n || x[sp] >= 0 || st < 0 || st >= vocab)) return -2;
    int r = run_inner(x, n, sp, st);
    if (r < 0 || status) {
      cleanup();
      return status == 1 ? -1 : (r < 0 ? r : -1);
    }
    return r;
  }

  // a gap node after the span in the frontier: a pending lexeme some byte
  // can extend stays open (epsilon), one no byte can extend emits its terminal
  __device__ int gap_from_frontier() {
    int c = open_column();
    if (c < 0) return -1;
    for (int f = 0; f < nf; ++f) {
      int q = ws.f_q[f];
      int a = g.dfa_accept[q];
      if (q == 0 || g.dfa_ext[q] || (a >= 0 && g.skip[a])) {
        arrive(ws.f_c[f], nullptr, false);
      } else if (a >= 0) {
        label_one(a);
        arrive(ws.f_c[f], sh.lbl, true);
      }
    }
    return c;
  }
  // the END node: the pending lexeme is flushed
  __device__ int end_from_frontier() {
    int c = open_column();
    if (c < 0) return -1;
    for (int f = 0; f < nf; ++f) {
      int q = ws.f_q[f];
      int a = g.dfa_accept[q];
      if (q == 0 || (a >= 0 && g.skip[a])) {
        arrive(ws.f_c[f], nullptr, false);
      } else if (a >= 0) {
        label_one(a);
        arrive(ws.f_c[f], sh.lbl, true);
      }
    }
    return c;
  }
  // frontier of a span that starts at column src: q0 at the sequence start,
  // every lexer state after a gap
  __device__ void frontier_from(int src, bool at_begin) {
    if (at_begin) {
      if (wl_lane() == 0) {
        ws.f_q[0] = 0;
        ws.f_c[0] = src;
      }
      nf = 1;
    } else {
      for (int q = wl_lane(); q < g.Q; q += 32) {
        ws.f_q[q] = q;
        ws.f_c[q] = src;
      }
      nf = g.Q;
    }
    __syncwarp();
  }
  __device__ void rec_range(int32_t* arr, int lo, int hi, int v) {
    for (int p = lo + (int)wl_lane(); p < hi; p += 32) arr[p] = v;
    __syncwarp();
  }

  __device__ int run_inner(const int32_t* x, int n, int sp, int stok) {
    int i = 0;
    bool first = true;
    int prev_gap = -1;
    int span_lo = -1, span_hi = -1;  // the last span, for post_col
    while (i < n) {
      int t0 = token_at(x, sp, stok, i);
      int j = i;
      if (t0 < 0) {
        while (j < n && token_at(x, sp, stok, j) < 0) ++j;
        int c;
        if (first) {
          c = open_column();
          if (c < 0) return -1;
          start_col = c;
          seed(c);
        } else {
          c = gap_from_frontier();
          if (c < 0) return -1;
        }
        close_column(c, true);
        finish_column(c);
        if (status) return -1;
        if (EXT && rec) {
          rec_range(rec->gap_col, i, j, c);
          if (span_lo >= 0) rec_range(rec->post_col, span_lo, span_hi, c);
        }
        prev_gap = c;
        if (column_empty(c)) return 0;
      } else {
        while (j < n && token_at(x, sp, stok, j) >= 0) ++j;
        int src;
        if (first) {
          int c = open_column();
          if (c < 0) return -1;
          start_col = c;
          seed(c);
          close_column(c, false);
          finish_column(c);
          if (status) return -1;
          src = c;
        } else {
          src = prev_gap;
        }
        frontier_from(src, first);
        if (EXT && rec) rec_range(rec->pre_col, i, j, src);
        span_lo = i;
        span_hi = j;
        for (int p = i; p < j && nf > 0; ++p) {
          int tok = token_at(x, sp, stok, p);
          if (tok < 0 || tok >= vocab) return -2;
          if (!span_step(tok)) return -1;
        }
        if (nf == 0) return 0;
        if (j == n) {  // END: flush the pending lexeme
          int c = end_from_frontier();
          if (c < 0) return -1;
          close_column(c, false);
          finish_column(c);
          if (status) return -1;
          if (EXT && rec) {
            rec_range(rec->post_col, i, j, c);
            if (wl_lane() == 0) rec->meta[3] = c;
          }
          return accepts(c, start_col) ? 1 : 0;
        }
      }
      first = false;
      i = j;
    }
    if (EXT && rec && wl_lane() == 0) rec->meta[3] = prev_gap;
    return accepts(prev_gap, start_col) ? 1 : 0;
  }
};

}  // namespace epic

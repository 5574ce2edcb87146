// Device-side data structures shared by the EPIC kernels.
#pragma once
#include <cstdint>

namespace epic {

// One lex-table entry (Sec. 4.1 / Alg. 2 memoization restated as a table):
// the greedy transducer's result for (token, entry state).
struct __align__(16) LexEntry {
  uint16_t end;     // end lexer state, 0xFFFF = DEAD
  uint8_t len;      // number of terminals emitted (skipped ones excluded)
  uint8_t term[13];
};
static_assert(sizeof(LexEntry) == 16, "lex entry is 16 bytes");

// Lazy lexing memo (Alg. 2's cache, filled on first use instead of built
// whole): an open-addressing table of (token, entry state) -> LexEntry.
// keys[h] = token * Q + state + 1 (0 = empty); ready[h] = 1 once vals[h] is
// written.  Null keys: the dense table is used.
struct LazyLex {
  uint32_t* keys;            // [cap]
  uint32_t* ready;           // [cap]
  LexEntry* vals;            // [cap]
  uint32_t mask;             // cap - 1 (cap a power of two)
  const int32_t* tok_off;    // [vocab + 1]
  const uint8_t* tok_bytes;
  unsigned long long* stats; // the table's counters: lookups, misses, computed without caching
};

// Grammar tables on the device (see grammar.h for their meaning).
struct DevGrammar {
  int T, V, D, W, VW, Q;
  int start_item, accept_item;
  const uint32_t* exp_term;       // [T][W]
  const uint32_t* exp_nt;         // [V][W]
  const uint32_t* any_nt;         // [W]
  const uint32_t* any_term;       // [W]
  const uint32_t* next_any;       // [W] items with a next symbol (excluding S' items)
  const uint32_t* nullable_next;  // [W]
  const uint32_t* complete;       // [W]
  const uint32_t* pred;           // [V][W]
  const uint32_t* gap_pred;       // [V][W]
  const int16_t* item_next;       // [D]
  const int16_t* item_lhs;        // [D]
  const int16_t* dfa_accept;      // [Q]
  const int32_t* dfa_next;        // [Q][256]
  const uint8_t* dfa_ext;         // [Q] 1 if some byte continues the lexeme
  const uint8_t* skip;            // [T]
  // advance closure by doubling: adv_pow[m][s][w] (m = 0: nullable_next,
  // m = 1: next_any) holds the items i with i .. i + 2^s - 1 all in the mask;
  // adv_steps doublings cover the longest production
  const uint32_t* adv_pow;        // [2][adv_steps][W]
  int adv_steps;
  // regular cover (flattened RTN), see cover.cuh
  int FS, FW;                     // cover states and words
  const uint32_t* cov_eps_close;  // [FS][FW] epsilon closure of each state
  const uint32_t* cov_all_close;  // [FS][FW] closure under every transition (a gap)
  const int32_t* cov_term_off;    // [T+1] CSR of labelled transitions by terminal
  const int32_t* cov_term_src;
  const int32_t* cov_term_dst;
  int cov_start, cov_accept;
  LazyLex lazy;                   // lexer tables built lazily (keys null: the dense table)
  // witness extraction: the complete items of each nonterminal (CSR over V)
  // and one shortest terminal string it derives (CSR over V)
  const int32_t* nt_comp_off;     // [V+1]
  const int32_t* nt_comp;
  const int32_t* ny_off;          // [V+1]
  const int32_t* ny;
  int gs_par;                     // CTA walks: warp-parallel origin sweep (gscols.cuh)
};

// The greedy transducer of one token from lexer state q (Sec. 4.1): at state
// s reading byte c, follow next(s, c) if defined; else, if s accepts, emit its
// terminal (unless skipped) and restart from next(q0, c); else DEAD.  Sets
// *overflow when the run exceeds 13 terminals (the entry is DEAD then).
__host__ __device__ inline LexEntry lex_transduce(const uint8_t* bytes, int b0, int b1, int q, const int32_t* dfa_next,
                                                  const int16_t* dfa_acc, const uint8_t* skip, bool* overflow) {
  LexEntry e;
  uint32_t* raw = reinterpret_cast<uint32_t*>(&e);
  raw[0] = raw[1] = raw[2] = raw[3] = 0;
  int s = q, len = 0;
  bool dead = false;
  for (int i = b0; i < b1; ++i) {
    const int c = bytes[i];
    const int nx = dfa_next[s * 256 + c];
    if (nx >= 0) {
      s = nx;
      continue;
    }
    const int a = dfa_acc[s];  // q0 never accepts (no terminal matches epsilon)
    if (a < 0) {
      dead = true;
      break;
    }
    if (!skip[a]) {
      if (len >= 13) {
        if (overflow) *overflow = true;
        dead = true;
        break;
      }
      e.term[len++] = (uint8_t)a;
    }
    s = dfa_next[c];  // restart from q0 on c
    if (s < 0) {
      dead = true;
      break;
    }
  }
  e.end = dead ? 0xFFFF : (uint16_t)s;
  e.len = dead ? 0 : (uint8_t)len;
  return e;
}

#ifdef __CUDACC__
// The lex entry of (token, state): from the dense table, or from the lazy
// memo, computing and inserting it on a miss.  Bounded: a full probe window
// (or a slot whose writer does not publish within the spin bound) computes
// the entry without caching it.
__device__ inline LexEntry lex_at(const DevGrammar& g, const LexEntry* table, int tok, int q) {
  if (!g.lazy.keys) return table[(size_t)tok * g.Q + q];
  const LazyLex& L = g.lazy;
  const uint32_t key = (uint32_t)tok * (uint32_t)g.Q + (uint32_t)q + 1u;
  uint32_t h = (key * 0x9E3779B1u) & L.mask;
  for (int probe = 0; probe < 64; ++probe, h = (h + 1) & L.mask) {
    uint32_t k = *((volatile const uint32_t*)&L.keys[h]);
    if (k == 0) {
      k = atomicCAS(&L.keys[h], 0u, key);
      if (k == 0) {  // this thread owns the slot: compute and publish
        const LexEntry e = lex_transduce(L.tok_bytes, L.tok_off[tok], L.tok_off[tok + 1], q, g.dfa_next,
                                         g.dfa_accept, g.skip, nullptr);
        L.vals[h] = e;
        __threadfence();
        atomicExch(&L.ready[h], 1u);
        atomicAdd(&L.stats[1], 1ull);
        return e;
      }
    }
    if (k == key) {
      // published by its owner, possibly a lane of this warp on another
      // branch: sleep between polls so that it runs
      for (int spin = 0; spin < (1 << 16); ++spin, __nanosleep(32))
        if (*((volatile const uint32_t*)&L.ready[h])) {
          __threadfence();
          const volatile uint32_t* v = reinterpret_cast<const volatile uint32_t*>(&L.vals[h]);
          LexEntry e;
          uint32_t* raw = reinterpret_cast<uint32_t*>(&e);
          raw[0] = v[0];
          raw[1] = v[1];
          raw[2] = v[2];
          raw[3] = v[3];
          return e;
        }
      break;  // not published in time: compute without the memo
    }
  }
  atomicAdd(&L.stats[2], 1ull);
  return lex_transduce(L.tok_bytes, L.tok_off[tok], L.tok_off[tok + 1], q, g.dfa_next, g.dfa_accept, g.skip, nullptr);
}
#endif

// Per-CTA workspace of the Earley walk (global memory).
struct Workspace {
  uint32_t* stage;   // [nmax][W] dense rows of the column under construction (zero when idle)
  uint32_t* bdone;   // [nmax][VW] nonterminals already completed per origin (current column)
  int32_t* col_off;  // [nmax + 1] entry range of each finished column
  int32_t* org;      // [emax] origin column of each entry
  uint32_t* bits;    // [emax][W]
  uint32_t* cov;     // [nmax][FW] cover state sets (selection kernels)
};

struct WsDims {
  int nmax;          // columns per check
  long long emax;    // entries per check
};

}  // namespace epic

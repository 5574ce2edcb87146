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
};

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

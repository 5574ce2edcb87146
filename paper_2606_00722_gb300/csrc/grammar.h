// Host-side grammar and lexer compilation for the EPIC hot path.
//
// epic_grammar_create turns a terminal/production description into the
// device tables the kernels use: a minimized union lexer DFA (terminal
// priority = lowest index), the dotted-item numbering of the CFG and the
// bitset masks that drive bit-parallel Earley recognition (Alg. 3) and the
// flattened regular cover (Sec. 4.3, App. A.2).
#pragma once
#include <cstdint>
#include <string>
#include <vector>

namespace epic {

constexpr int kMaxRhs = 62;           // dotted positions fit in 6 bits
constexpr int kMaxRun = 13;           // terminals per lex-table entry
constexpr int kLexDead = 0xFFFF;      // end-state value of a DEAD entry

struct LexerDFA {
  int Q = 0;                          // states; state 0 is the initial state q0
  std::vector<int32_t> next;          // [Q][256], -1 = no transition
  std::vector<int16_t> accept;        // [Q] terminal accepted (lowest index), -1 = none
};

// Glushkov construction per terminal regex, subset construction of the union,
// Moore minimization.  Throws std::runtime_error on malformed input or on a
// terminal that matches the empty string.
LexerDFA build_lexer(const std::vector<std::string>& regex);

struct GrammarTables {
  int T = 0, V = 0, P = 0, start = 0;   // after trimming: symbols keep their ids
  std::vector<uint8_t> skip;            // [T]
  std::vector<uint8_t> term_used;       // [T] terminal occurs in a kept rhs
  // productions kept after trimming, plus the augmented S' -> S (last)
  std::vector<int32_t> lhs;             // [P'] (-1 for S')
  std::vector<int32_t> rhs_off, rhs;    // CSR
  int aug = -1;
  // dotted items: item(p, d) = item_base[p] + d, d in 0..|rhs_p|
  int D = 0, W = 0;                     // items and 32-bit words per item bitset
  std::vector<int32_t> item_base;       // [P']
  std::vector<int32_t> item_next;       // [D] symbol after the dot, -1 if complete
  std::vector<int32_t> item_lhs;        // [D] lhs of the item's production (-1 for S')
  std::vector<uint8_t> nullable;        // [V]
  // masks, each W words
  std::vector<uint32_t> exp_term;       // [T][W] items whose next symbol is terminal a
  std::vector<uint32_t> exp_nt;         // [V][W] items whose next symbol is NT B
  std::vector<uint32_t> any_term;       // [W]
  std::vector<uint32_t> any_nt;         // [W]
  std::vector<uint32_t> nullable_next;  // [W] next symbol is a nullable NT
  std::vector<uint32_t> complete;       // [W] complete items (excluding S')
  std::vector<uint32_t> pred;           // [V][W] Earley prediction closure of B
  std::vector<uint32_t> gap_pred;       // [V][W] items predicted and fully advanced inside a gap
  int accept_item = -1;                 // S' -> S .
  int start_item = -1;                  // S' -> . S
};

GrammarTables build_tables(int T, const std::vector<uint8_t>& skip, int V, int start,
                           const std::vector<int32_t>& lhs, const std::vector<int32_t>& rhs_off,
                           const std::vector<int32_t>& rhs);

}  // namespace epic

namespace epic {
// Flattened RTN regular cover of the trimmed grammar (Sec. 4.3, App. A.2):
// states 0..D-1 are the dotted items, D + A is entry(A), D + V + A is exit(A).
struct CoverTables {
  int FS = 0, FW = 0, start = 0, accept = 0;
  std::vector<uint32_t> eps_close;  // [FS][FW] closure under epsilon edges
  std::vector<uint32_t> all_close;  // [FS][FW] closure under every edge
};
CoverTables build_cover(const GrammarTables& G);
}  // namespace epic

// Host-side grammar and lexer compilation (see grammar.h).
#include "grammar.h"

#include <algorithm>
#include <map>
#include <memory>
#include <set>
#include <stdexcept>

namespace epic {
namespace {

// ---------------------------------------------------------------- regex AST
struct Node {
  enum Kind { Leaf, Cat, Alt, Star, Plus, Opt, Empty } kind;
  std::unique_ptr<Node> a, b;
  int pos = -1;  // leaf: global position id
};
using NodeP = std::unique_ptr<Node>;

struct Pos {
  uint32_t cls[8] = {0};  // 256-bit byte class
  int term = 0;
  bool has(int c) const { return (cls[c >> 5] >> (c & 31)) & 1u; }
};

// Tokenizing recursive-descent parser over the syntax documented in epic.h.
class Parser {
 public:
  Parser(const std::string& src, int term, std::vector<Pos>& pos) : s_(src), term_(term), pos_(pos) {}
  NodeP parse() {
    NodeP n = alternation();
    if (i_ != s_.size()) fail("unbalanced ')'");
    return n;
  }

 private:
  const std::string& s_;
  size_t i_ = 0;
  int term_;
  std::vector<Pos>& pos_;

  [[noreturn]] void fail(const char* why) {
    throw std::runtime_error(std::string("terminal regex: ") + why);
  }
  static NodeP make(Node::Kind k, NodeP a = nullptr, NodeP b = nullptr) {
    NodeP n(new Node{k, std::move(a), std::move(b)});
    return n;
  }
  NodeP leaf(const Pos& p) {
    NodeP n = make(Node::Leaf);
    n->pos = (int)pos_.size();
    pos_.push_back(p);
    pos_.back().term = term_;
    return n;
  }
  int esc() {
    if (i_ >= s_.size()) fail("escape at end");
    char c = s_[i_++];
    switch (c) {
      case 'n': return '\n';
      case 't': return '\t';
      case 'r': return '\r';
      default: return (unsigned char)c;
    }
  }
  NodeP alternation() {
    NodeP left = concatenation();
    while (i_ < s_.size() && s_[i_] == '|') {
      ++i_;
      left = make(Node::Alt, std::move(left), concatenation());
    }
    return left;
  }
  NodeP concatenation() {
    NodeP acc;
    while (i_ < s_.size() && s_[i_] != '|' && s_[i_] != ')') {
      NodeP f = postfix();
      acc = acc ? make(Node::Cat, std::move(acc), std::move(f)) : std::move(f);
    }
    return acc ? std::move(acc) : make(Node::Empty);
  }
  NodeP postfix() {
    NodeP n = primary();
    for (;;) {
      if (i_ >= s_.size()) break;
      char c = s_[i_];
      if (c == '*')
        n = make(Node::Star, std::move(n));
      else if (c == '+')
        n = make(Node::Plus, std::move(n));
      else if (c == '?')
        n = make(Node::Opt, std::move(n));
      else
        break;
      ++i_;
    }
    return n;
  }
  NodeP primary() {
    if (i_ >= s_.size()) fail("unexpected end");
    char c = s_[i_++];
    Pos p;
    auto set = [&](int v) { p.cls[v >> 5] |= 1u << (v & 31); };
    switch (c) {
      case '(': {
        NodeP n = alternation();
        if (i_ >= s_.size() || s_[i_] != ')') fail("missing ')'");
        ++i_;
        return n;
      }
      case '[': {
        bool neg = (i_ < s_.size() && s_[i_] == '^');
        if (neg) ++i_;
        bool done = false;
        while (i_ < s_.size()) {
          char d = s_[i_++];
          if (d == ']') {
            done = true;
            break;
          }
          int lo = d == '\\' ? esc() : (unsigned char)d, hi = lo;
          if (i_ + 1 < s_.size() && s_[i_] == '-' && s_[i_ + 1] != ']') {
            ++i_;
            char e = s_[i_++];
            hi = e == '\\' ? esc() : (unsigned char)e;
          }
          if (hi < lo) fail("reversed class range");
          for (int v = lo; v <= hi; ++v) set(v);
        }
        if (!done) fail("missing ']'");
        if (neg)
          for (int w = 0; w < 8; ++w) p.cls[w] = ~p.cls[w];
        return leaf(p);
      }
      case '.':
        for (int v = 0; v < 256; ++v)
          if (v != '\n') set(v);
        return leaf(p);
      case '\\':
        set(esc());
        return leaf(p);
      case ')': case '*': case '+': case '?': case ']':
        fail("operator without operand");
      default:
        set((unsigned char)c);
        return leaf(p);
    }
  }
};

// Glushkov sets of a subtree.
struct Gl {
  bool nullable;
  std::vector<int> first, last;
};

std::vector<int> merge(const std::vector<int>& a, const std::vector<int>& b) {
  std::vector<int> r;
  std::set_union(a.begin(), a.end(), b.begin(), b.end(), std::back_inserter(r));
  return r;
}

Gl glushkov(const Node* n, std::vector<std::vector<int>>& follow) {
  auto link = [&](const std::vector<int>& from, const std::vector<int>& to) {
    for (int p : from) follow[p] = merge(follow[p], to);
  };
  switch (n->kind) {
    case Node::Leaf: return {false, {n->pos}, {n->pos}};
    case Node::Empty: return {true, {}, {}};
    case Node::Cat: {
      Gl a = glushkov(n->a.get(), follow), b = glushkov(n->b.get(), follow);
      link(a.last, b.first);
      return {a.nullable && b.nullable, a.nullable ? merge(a.first, b.first) : a.first,
              b.nullable ? merge(a.last, b.last) : b.last};
    }
    case Node::Alt: {
      Gl a = glushkov(n->a.get(), follow), b = glushkov(n->b.get(), follow);
      return {a.nullable || b.nullable, merge(a.first, b.first), merge(a.last, b.last)};
    }
    case Node::Star:
    case Node::Plus:
    case Node::Opt: {
      Gl a = glushkov(n->a.get(), follow);
      if (n->kind != Node::Opt) link(a.last, a.first);
      return {a.nullable || n->kind != Node::Plus, a.first, a.last};
    }
  }
  return {true, {}, {}};
}

}  // namespace

LexerDFA build_lexer(const std::vector<std::string>& regex) {
  std::vector<Pos> pos;
  std::vector<NodeP> roots;
  for (size_t t = 0; t < regex.size(); ++t) roots.push_back(Parser(regex[t], (int)t, pos).parse());
  std::vector<std::vector<int>> follow(pos.size());
  std::vector<int> first_all;
  std::vector<char> is_last(pos.size(), 0);
  for (size_t t = 0; t < roots.size(); ++t) {
    Gl g = glushkov(roots[t].get(), follow);
    if (g.nullable) throw std::runtime_error("terminal " + std::to_string(t) + " matches the empty string");
    first_all = merge(first_all, g.first);
    for (int p : g.last) is_last[p] = 1;
  }
  // subset construction; a state is the set of positions just matched, the
  // initial state is the empty set
  std::map<std::vector<int>, int> id;
  std::vector<std::vector<int>> states{{}};
  id[{}] = 0;
  std::vector<int32_t> next;
  std::vector<int16_t> acc;
  for (size_t s = 0; s < states.size(); ++s) {
    const std::vector<int> cur = states[s];
    std::vector<int> cand = first_all;
    if (!cur.empty()) {
      cand.clear();
      for (int p : cur) cand = merge(cand, follow[p]);
    }
    int best = -1;
    for (int p : cur)
      if (is_last[p] && (best < 0 || pos[p].term < best)) best = pos[p].term;
    acc.push_back((int16_t)best);
    for (int c = 0; c < 256; ++c) {
      std::vector<int> to;
      for (int p : cand)
        if (pos[p].has(c)) to.push_back(p);
      if (to.empty()) {
        next.push_back(-1);
        continue;
      }
      auto it = id.find(to);
      int t;
      if (it == id.end()) {
        t = (int)states.size();
        id[to] = t;
        states.push_back(to);
      } else {
        t = it->second;
      }
      next.push_back(t);
    }
  }
  // Moore minimization: blocks start by accepted terminal, refine on the
  // blocks of the 256 successors (no transition is its own block).
  int n = (int)states.size();
  std::vector<int> blk(n);
  {
    std::map<int, int> by_acc;
    for (int s = 0; s < n; ++s) {
      auto it = by_acc.emplace(acc[s], (int)by_acc.size()).first;
      blk[s] = it->second;
    }
  }
  for (;;) {
    std::map<std::vector<int>, int> sig_id;
    std::vector<int> nb(n);
    for (int s = 0; s < n; ++s) {
      std::vector<int> sig;
      sig.reserve(257);
      sig.push_back(blk[s]);
      for (int c = 0; c < 256; ++c) sig.push_back(next[s * 256 + c] < 0 ? -1 : blk[next[s * 256 + c]]);
      nb[s] = sig_id.emplace(sig, (int)sig_id.size()).first->second;
    }
    bool same = sig_id.size() == std::set<int>(blk.begin(), blk.end()).size();
    blk = nb;
    if (same) break;
  }
  // renumber so that the initial state's block is 0, others by first appearance
  std::vector<int> ren(n, -1);
  int Q = 0;
  for (int s = 0; s < n; ++s)
    if (ren[blk[s]] < 0) ren[blk[s]] = Q++;
  LexerDFA dfa;
  dfa.Q = Q;
  dfa.next.assign((size_t)Q * 256, -1);
  dfa.accept.assign(Q, -1);
  for (int s = 0; s < n; ++s) {
    int q = ren[blk[s]];
    dfa.accept[q] = acc[s];
    for (int c = 0; c < 256; ++c)
      dfa.next[(size_t)q * 256 + c] = next[s * 256 + c] < 0 ? -1 : ren[blk[next[s * 256 + c]]];
  }
  return dfa;
}

GrammarTables build_tables(int T, const std::vector<uint8_t>& skip, int V, int start,
                           const std::vector<int32_t>& lhs, const std::vector<int32_t>& rhs_off,
                           const std::vector<int32_t>& rhs) {
  GrammarTables G;
  G.T = T;
  G.V = V;
  G.start = start;
  G.skip = skip;
  int P = (int)lhs.size();
  if (start < 0 || start >= V) throw std::invalid_argument("start symbol out of range");
  for (int p = 0; p < P; ++p) {
    if (lhs[p] < 0 || lhs[p] >= V) throw std::invalid_argument("lhs out of range");
    if (rhs_off[p + 1] < rhs_off[p]) throw std::invalid_argument("rhs_off not monotone");
    if (rhs_off[p + 1] - rhs_off[p] > kMaxRhs) throw std::invalid_argument("rhs too long");
    for (int i = rhs_off[p]; i < rhs_off[p + 1]; ++i) {
      int s = rhs[i];
      if (s < 0 || s >= T + V) throw std::invalid_argument("rhs symbol out of range");
      if (s < T && skip[s]) throw std::invalid_argument("skipped terminal used in a production");
    }
  }
  // trim: productive symbols, then reachable from the start
  std::vector<char> prod(V, 0);
  for (bool ch = true; ch;) {
    ch = false;
    for (int p = 0; p < P; ++p) {
      if (prod[lhs[p]]) continue;
      bool ok = true;
      for (int i = rhs_off[p]; i < rhs_off[p + 1] && ok; ++i)
        if (rhs[i] >= T && !prod[rhs[i] - T]) ok = false;
      if (ok) prod[lhs[p]] = ch = true;
    }
  }
  if (!prod[start]) throw std::domain_error("the grammar's language is empty");
  auto usable = [&](int p) {
    if (!prod[lhs[p]]) return false;
    for (int i = rhs_off[p]; i < rhs_off[p + 1]; ++i)
      if (rhs[i] >= T && !prod[rhs[i] - T]) return false;
    return true;
  };
  std::vector<char> reach(V, 0);
  reach[start] = 1;
  for (bool ch = true; ch;) {
    ch = false;
    for (int p = 0; p < P; ++p)
      if (reach[lhs[p]] && usable(p))
        for (int i = rhs_off[p]; i < rhs_off[p + 1]; ++i)
          if (rhs[i] >= T && !reach[rhs[i] - T]) reach[rhs[i] - T] = ch = true;
  }
  G.rhs_off.push_back(0);
  G.term_used.assign(T, 0);
  for (int p = 0; p < P; ++p) {
    if (!reach[lhs[p]] || !usable(p)) continue;
    G.lhs.push_back(lhs[p]);
    for (int i = rhs_off[p]; i < rhs_off[p + 1]; ++i) {
      G.rhs.push_back(rhs[i]);
      if (rhs[i] < T) G.term_used[rhs[i]] = 1;
    }
    G.rhs_off.push_back((int)G.rhs.size());
  }
  G.aug = (int)G.lhs.size();
  G.lhs.push_back(-1);
  G.rhs.push_back(T + start);
  G.rhs_off.push_back((int)G.rhs.size());
  G.P = (int)G.lhs.size();
  // nullable nonterminals
  G.nullable.assign(V, 0);
  for (bool ch = true; ch;) {
    ch = false;
    for (int p = 0; p < G.aug; ++p) {
      if (G.nullable[G.lhs[p]]) continue;
      bool ok = true;
      for (int i = G.rhs_off[p]; i < G.rhs_off[p + 1] && ok; ++i)
        ok = G.rhs[i] >= T && G.nullable[G.rhs[i] - T];
      if (ok) G.nullable[G.lhs[p]] = ch = true;
    }
  }
  // items
  G.item_base.resize(G.P);
  int D = 0;
  for (int p = 0; p < G.P; ++p) {
    G.item_base[p] = D;
    D += G.rhs_off[p + 1] - G.rhs_off[p] + 1;
  }
  G.D = D;
  G.W = (D + 31) / 32;
  int W = G.W;
  G.item_next.assign(D, -1);
  G.item_lhs.assign(D, -1);
  for (int p = 0; p < G.P; ++p) {
    int len = G.rhs_off[p + 1] - G.rhs_off[p];
    for (int d = 0; d <= len; ++d) {
      G.item_lhs[G.item_base[p] + d] = G.lhs[p];
      if (d < len) G.item_next[G.item_base[p] + d] = G.rhs[G.rhs_off[p] + d];
    }
  }
  G.start_item = G.item_base[G.aug];
  G.accept_item = G.start_item + 1;
  auto setb = [&](std::vector<uint32_t>& m, size_t off, int i) { m[off + (i >> 5)] |= 1u << (i & 31); };
  G.exp_term.assign((size_t)T * W, 0);
  G.exp_nt.assign((size_t)V * W, 0);
  G.any_term.assign(W, 0);
  G.any_nt.assign(W, 0);
  G.nullable_next.assign(W, 0);
  G.complete.assign(W, 0);
  for (int i = 0; i < D; ++i) {
    int X = G.item_next[i];
    if (X < 0) {
      if (i != G.accept_item) setb(G.complete, 0, i);
    } else if (X < T) {
      setb(G.exp_term, (size_t)X * W, i);
      setb(G.any_term, 0, i);
    } else {
      setb(G.exp_nt, (size_t)(X - T) * W, i);
      setb(G.any_nt, 0, i);
      if (G.nullable[X - T]) setb(G.nullable_next, 0, i);
    }
  }
  std::vector<std::vector<int>> prods_of(V);
  for (int p = 0; p < G.aug; ++p) prods_of[G.lhs[p]].push_back(p);
  // Earley prediction closure of B, with the dot already advanced over
  // nullable prefixes (Aycock & Horspool): the left-corner closure.
  G.pred.assign((size_t)V * W, 0);
  G.gap_pred.assign((size_t)V * W, 0);
  for (int B = 0; B < V; ++B) {
    std::vector<char> in(V, 0), in_all(V, 0);
    std::vector<int> st{B};
    in[B] = 1;
    while (!st.empty()) {
      int A = st.back();
      st.pop_back();
      for (int p : prods_of[A]) {
        for (int i = G.rhs_off[p]; i < G.rhs_off[p + 1]; ++i) {
          int d = i - G.rhs_off[p];
          setb(G.pred, (size_t)B * W, G.item_base[p] + d);
          int X = G.rhs[i];
          if (X < T) break;
          if (!in[X - T]) {
            in[X - T] = 1;
            st.push_back(X - T);
          }
          if (!G.nullable[X - T]) break;
          if (i + 1 == G.rhs_off[p + 1]) setb(G.pred, (size_t)B * W, G.item_base[p] + d + 1);
        }
        if (G.rhs_off[p] == G.rhs_off[p + 1]) setb(G.pred, (size_t)B * W, G.item_base[p]);
      }
    }
    // inside a gap every symbol derives some string of Sigma_lex*, so all
    // items of every nonterminal reachable from B appear
    st.push_back(B);
    in_all[B] = 1;
    while (!st.empty()) {
      int A = st.back();
      st.pop_back();
      for (int p : prods_of[A]) {
        int len = G.rhs_off[p + 1] - G.rhs_off[p];
        for (int d = 0; d <= len; ++d) setb(G.gap_pred, (size_t)B * W, G.item_base[p] + d);
        for (int i = G.rhs_off[p]; i < G.rhs_off[p + 1]; ++i) {
          int X = G.rhs[i];
          if (X >= T && !in_all[X - T]) {
            in_all[X - T] = 1;
            st.push_back(X - T);
          }
        }
      }
    }
  }
  return G;
}

}  // namespace epic

namespace epic {

CoverTables build_cover(const GrammarTables& G) {
  CoverTables C;
  int D = G.D, V = G.V, T = G.T;
  C.FS = D + 2 * V;
  C.FW = (C.FS + 31) / 32;
  C.start = D + G.start;
  C.accept = D + V + G.start;
  std::vector<std::vector<int>> eps(C.FS), lab(C.FS);
  for (int p = 0; p < G.aug; ++p) {
    int A = G.lhs[p];
    int base = G.item_base[p];
    int len = G.rhs_off[p + 1] - G.rhs_off[p];
    eps[D + A].push_back(base);                 // entry(A) -> (p, 0)
    for (int d = 0; d < len; ++d) {
      int X = G.rhs[G.rhs_off[p] + d];
      if (X < T) {
        lab[base + d].push_back(base + d + 1);  // (p, d) -a-> (p, d+1)
      } else {
        eps[base + d].push_back(D + (X - T));   // call: (p, d) -> entry(B)
        eps[D + V + (X - T)].push_back(base + d + 1);  // return: exit(B) -> (p, d+1)
      }
    }
    eps[base + len].push_back(D + V + A);       // (p, |rhs|) -> exit(A)
  }
  auto close = [&](bool all, std::vector<uint32_t>& out) {
    out.assign((size_t)C.FS * C.FW, 0);
    std::vector<int> stack;
    std::vector<char> seen(C.FS);
    for (int s = 0; s < C.FS; ++s) {
      std::fill(seen.begin(), seen.end(), 0);
      stack.assign(1, s);
      seen[s] = 1;
      while (!stack.empty()) {
        int u = stack.back();
        stack.pop_back();
        out[(size_t)s * C.FW + (u >> 5)] |= 1u << (u & 31);
        for (int v : eps[u])
          if (!seen[v]) { seen[v] = 1; stack.push_back(v); }
        if (all)
          for (int v : lab[u])
            if (!seen[v]) { seen[v] = 1; stack.push_back(v); }
      }
    }
  };
  close(false, C.eps_close);
  close(true, C.all_close);
  return C;
}

}  // namespace epic

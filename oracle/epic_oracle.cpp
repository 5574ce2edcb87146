// EPIC validity oracle -- TEST INFRASTRUCTURE ONLY.
//
// A plain, slow, single-purpose CPU implementation of what the hot path
// computes, written from the paper (arXiv 2606.00722, "EPIC: Efficient and
// Parallel Inference under CFG Constraints for Diffusion Language Models"):
//
//   * Valid_G(x, Delta) = 1[ L(G) cap C_{x (+) Delta} != empty ]   (Sec. 3)
//     with (x (+) Delta) applied position-wise                      (Sec. 3)
//   * C_x = L(A_x), the epsilon-NFA of compatible lexeme sequences  (Sec. 3, Alg. 2)
//   * the Earley-style graph parser deciding it                     (Alg. 3, App. C.3)
//   * the flattened recursive-transition-network regular cover      (Sec. 4.3, App. A.2, App. D.3)
//   * relaxed compatible subset selection + exact shrink            (Alg. 4)
//   * the sequential rejection fallback                             (Alg. 1)
//   * membership of a terminal string in a partial output's graph   (witness checks, Sec. 4.4)
//
// Where the paper is silent (lexer rule, gap model, cover flattening,
// tie-breaks) a reading is taken; each is stated where it is implemented
// below.
//
// Only tests, the smoke check and the benchmark's CPU-baseline leg and
// reference arm may load this library.  It shares no code, header or table with the CUDA path: it
// has its own regex parser, its own lexer (per-terminal Thompson NFAs run by
// subset simulation, no DFA tables), its own graph and its own parser.
#include <algorithm>
#include <atomic>
#include <cstdint>
#include <cstring>
#include <map>
#include <set>
#include <stdexcept>
#include <string>
#include <thread>
#include <tuple>
#include <unordered_map>
#include <unordered_set>
#include <vector>

namespace {

// ------------------------------------------------------------------ regex
// Thompson construction.  One NFA per terminal, all states in one pool.
struct NState {
  std::vector<std::pair<std::vector<bool>, int>> moves;  // (byte set, target)
  std::vector<int> eps;
  int accept_term = -1;                                  // terminal accepted here
};

struct Frag {
  int start, accept;
};

struct RegexParser {
  std::vector<NState>& pool;
  const std::string s;
  size_t i = 0;
  RegexParser(std::vector<NState>& p, const std::string& src) : pool(p), s(src) {}

  int fresh() {
    pool.emplace_back();
    return (int)pool.size() - 1;
  }
  Frag byteset(const std::vector<bool>& set) {
    int a = fresh(), b = fresh();
    pool[a].moves.push_back({set, b});
    return {a, b};
  }
  Frag eps_frag() {
    int a = fresh(), b = fresh();
    pool[a].eps.push_back(b);
    return {a, b};
  }
  int escaped_byte() {
    if (i >= s.size()) throw std::runtime_error("dangling escape");
    char c = s[i++];
    if (c == 'n') return '\n';
    if (c == 't') return '\t';
    if (c == 'r') return '\r';
    return (unsigned char)c;
  }
  Frag parse_alt() {
    Frag f = parse_concat();
    while (i < s.size() && s[i] == '|') {
      ++i;
      Frag g = parse_concat();
      int a = fresh(), b = fresh();
      pool[a].eps.push_back(f.start);
      pool[a].eps.push_back(g.start);
      pool[f.accept].eps.push_back(b);
      pool[g.accept].eps.push_back(b);
      f = {a, b};
    }
    return f;
  }
  Frag parse_concat() {
    bool any = false;
    Frag f{-1, -1};
    while (i < s.size() && s[i] != '|' && s[i] != ')') {
      Frag g = parse_repeat();
      if (!any) {
        f = g;
        any = true;
      } else {
        pool[f.accept].eps.push_back(g.start);
        f.accept = g.accept;
      }
    }
    return any ? f : eps_frag();
  }
  Frag parse_repeat() {
    Frag f = parse_atom();
    while (i < s.size() && (s[i] == '*' || s[i] == '+' || s[i] == '?')) {
      char op = s[i++];
      int a = fresh(), b = fresh();
      pool[a].eps.push_back(f.start);
      pool[f.accept].eps.push_back(b);
      if (op == '*' || op == '?') pool[a].eps.push_back(b);
      if (op == '*' || op == '+') pool[f.accept].eps.push_back(f.start);
      f = {a, b};
    }
    return f;
  }
  Frag parse_atom() {
    if (i >= s.size()) throw std::runtime_error("unexpected end of regex");
    char c = s[i++];
    if (c == '(') {
      Frag f = parse_alt();
      if (i >= s.size() || s[i] != ')') throw std::runtime_error("missing )");
      ++i;
      return f;
    }
    std::vector<bool> set(256, false);
    if (c == '[') {
      bool neg = false;
      if (i < s.size() && s[i] == '^') {
        neg = true;
        ++i;
      }
      bool closed = false;
      while (i < s.size()) {
        char d = s[i++];
        if (d == ']') {
          closed = true;
          break;
        }
        int lo = (d == '\\') ? escaped_byte() : (unsigned char)d;
        int hi = lo;
        if (i + 1 < s.size() && s[i] == '-' && s[i + 1] != ']') {
          ++i;
          char e = s[i++];
          hi = (e == '\\') ? escaped_byte() : (unsigned char)e;
        }
        if (hi < lo) throw std::runtime_error("bad class range");
        for (int v = lo; v <= hi; ++v) set[v] = true;
      }
      if (!closed) throw std::runtime_error("missing ]");
      if (neg)
        for (int v = 0; v < 256; ++v) set[v] = !set[v];
      return byteset(set);
    }
    if (c == ')' || c == '*' || c == '+' || c == '?' || c == ']')
      throw std::runtime_error("unexpected regex operator");
    if (c == '.') {
      for (int v = 0; v < 256; ++v) set[v] = (v != '\n');
      return byteset(set);
    }
    int v = (c == '\\') ? escaped_byte() : (unsigned char)c;
    set[v] = true;
    return byteset(set);
  }
};

// ------------------------------------------------------------------ grammar
struct Grammar {
  int T = 0, V = 0, start = 0;
  std::vector<bool> skip;
  std::vector<int> lhs;                  // per production (augmented prod last)
  std::vector<std::vector<int>> rhs;     // symbols: <T terminal, >=T nonterminal
  std::vector<std::vector<int>> prods_of;  // NT -> productions
  int aug = -1;                          // S' -> S
  // lexer
  std::vector<NState> nfa;
  std::vector<int> term_start;
  std::vector<int> q0;                   // closure of all starts (sorted)
  std::map<std::vector<int>, int> state_id;  // live lexer states
  std::vector<std::vector<int>> states;
  // vocab
  std::vector<std::string> vocab;
  std::string error;
};

std::vector<int> eclose(const Grammar& g, std::vector<int> set) {
  std::vector<char> seen(g.nfa.size(), 0);
  std::vector<int> stack = set, out;
  for (int s : set) seen[s] = 1;
  while (!stack.empty()) {
    int s = stack.back();
    stack.pop_back();
    out.push_back(s);
    for (int t : g.nfa[s].eps)
      if (!seen[t]) {
        seen[t] = 1;
        stack.push_back(t);
      }
  }
  std::sort(out.begin(), out.end());
  return out;
}

std::vector<int> step(const Grammar& g, const std::vector<int>& q, int c) {
  std::vector<int> nxt;
  for (int s : q)
    for (auto& mv : g.nfa[s].moves)
      if (mv.first[c]) nxt.push_back(mv.second);
  if (nxt.empty()) return nxt;
  std::sort(nxt.begin(), nxt.end());
  nxt.erase(std::unique(nxt.begin(), nxt.end()), nxt.end());
  return eclose(g, nxt);
}

// lowest-index terminal accepted by the state set, or -1
int accepts(const Grammar& g, const std::vector<int>& q) {
  int best = -1;
  for (int s : q)
    if (g.nfa[s].accept_term >= 0 && (best < 0 || g.nfa[s].accept_term < best))
      best = g.nfa[s].accept_term;
  return best;
}

// true if some byte continues the lexeme in state q
bool extensible(const Grammar& g, const std::vector<int>& q) {
  for (int c = 0; c < 256; ++c)
    if (!step(g, q, c).empty()) return true;
  return false;
}

// Greedy lexing transducer (reading of the lexical map; the paper delegates
// lexing to prior work): at state q reading byte c, continue if a transition
// exists; otherwise, if q accepts (q != q0), emit its terminal and restart
// from q0 on c; otherwise the lexing dies.  At the end of the sequence a q0
// state emits nothing, an accepting state emits its terminal, anything else
// dies.  Before a gap (flush_end false) the pending lexeme stays open when
// some byte could extend it (the gap absorbs its terminal); a lexeme that no
// byte can extend has ended, so an accepting state emits its terminal.
// Skipped terminals are dropped from the run.  Returns false on DEAD.
enum LexEnd { kRunOnly = 0, kEndFlush = 1, kBeforeGap = 2 };

bool lex_run_mode(const Grammar& g, const std::vector<int>& entry, const std::string& bytes, int mode,
                  std::vector<int>& run, std::vector<int>& pending);

bool lex_run(const Grammar& g, const std::vector<int>& entry, const std::string& bytes,
             bool flush_end, std::vector<int>& run, std::vector<int>& pending) {
  return lex_run_mode(g, entry, bytes, flush_end ? kEndFlush : kBeforeGap, run, pending);
}

bool lex_run_mode(const Grammar& g, const std::vector<int>& entry, const std::string& bytes, int mode,
                  std::vector<int>& run, std::vector<int>& pending) {
  bool flush_end = mode == kEndFlush;
  std::vector<int> q = entry;
  run.clear();
  for (unsigned char c : bytes) {
    std::vector<int> n = step(g, q, c);
    if (!n.empty()) {
      q.swap(n);
      continue;
    }
    int t = accepts(g, q);
    if (q == g.q0 || t < 0) return false;
    if (!g.skip[t]) run.push_back(t);
    q = step(g, g.q0, c);
    if (q.empty()) return false;
  }
  if (mode == kBeforeGap && q != g.q0 && !extensible(g, q)) {
    int t = accepts(g, q);
    if (t < 0) return false;
    if (!g.skip[t]) run.push_back(t);
    q = g.q0;
  }
  if (flush_end) {
    if (q != g.q0) {
      int t = accepts(g, q);
      if (t < 0) return false;
      if (!g.skip[t]) run.push_back(t);
    }
    q = g.q0;
  }
  pending = q;
  return true;
}

// ------------------------------------------------------------------ graph
// The epsilon-NFA A_x (Sec. 3, Alg. 2) for a partial output, under the gap
// reading: every maximal run of masks is one gap node with a self-loop on
// every terminal (Sigma_lex*); every maximal run of fixed tokens is a span
// whose distinct lexings become alternative paths between its neighbours.
// A span after a gap may start inside a lexeme begun in the gap, so it is
// lexed from every live lexer state; a span before a gap keeps its pending
// lexeme open into the gap when a byte could extend it (its terminal is
// absorbed by Sigma_lex*) and emits it otherwise; the last span of the
// sequence flushes at END.
struct Graph {
  int n_nodes = 0;
  std::vector<char> gap;
  std::vector<std::vector<std::pair<int, int>>> out;  // (label, target); label -1 = epsilon
  int start = 0, accept = 0;
  bool dead = false;                                   // some span has no lexing
};

int add_node(Graph& G, bool is_gap) {
  G.gap.push_back(is_gap ? 1 : 0);
  G.out.emplace_back();
  return G.n_nodes++;
}

// Alg. 2's cache: the alternatives of a span depend only on its bytes and
// its boundary condition (sequence start / after a gap, sequence end / before
// a gap), so they are memoized under that key; the graph is unchanged.
using LexMemo = std::map<std::tuple<std::string, bool, bool>, std::set<std::vector<int>>>;

const std::set<std::vector<int>>& span_alternatives(const Grammar& g, LexMemo& memo,
                                                    const std::string& bytes, bool at_begin,
                                                    bool at_end) {
  auto key = std::make_tuple(bytes, at_begin, at_end);
  auto it = memo.find(key);
  if (it != memo.end()) return it->second;
  std::set<std::vector<int>> alts;
  std::vector<int> run, pend;
  if (at_begin) {
    if (lex_run(g, g.q0, bytes, at_end, run, pend)) alts.insert(run);
  } else {
    for (auto& e : g.states)  // every live lexer state
      if (lex_run(g, e, bytes, at_end, run, pend)) alts.insert(run);
  }
  return memo.emplace(key, std::move(alts)).first->second;
}

Graph build_graph(const Grammar& g, const std::vector<int>& x, LexMemo& memo) {
  Graph G;
  int n = (int)x.size();
  if (n == 0) {  // the empty output: valid iff epsilon is in L(G)
    G.start = G.accept = add_node(G, false);
    return G;
  }
  int cur = -1;
  int i = 0;
  bool first = true;
  while (i < n) {
    int j = i;
    if (x[i] < 0) {
      while (j < n && x[j] < 0) ++j;
      int gnode = add_node(G, true);
      if (cur < 0)
        G.start = gnode;
      else
        G.out[cur].push_back({-1, gnode});  // span already ended in cur
      cur = gnode;
    } else {
      while (j < n && x[j] >= 0) ++j;
      std::string bytes;
      for (int t = i; t < j; ++t) bytes += g.vocab[x[t]];
      bool at_begin = first;
      bool at_end = (j == n);
      const std::set<std::vector<int>>& alts = span_alternatives(g, memo, bytes, at_begin, at_end);
      int pred = cur;
      if (pred < 0) {
        pred = add_node(G, false);  // BEGIN
        G.start = pred;
      }
      if (alts.empty()) G.dead = true;
      // Alternatives share their common suffixes (a reversed trie rooted at
      // succ): the node reached after a run's first i terminals is keyed by
      // the remaining suffix, so the graph's language is the set of runs.
      // Nodes are numbered in topological order: pred, then the suffix nodes
      // by decreasing suffix length, then succ.
      std::set<std::vector<int>> suffixes;
      for (auto& r : alts)
        for (size_t t = 1; t < r.size(); ++t) suffixes.insert(std::vector<int>(r.begin() + t, r.end()));
      std::vector<std::vector<int>> order(suffixes.begin(), suffixes.end());
      std::stable_sort(order.begin(), order.end(),
                       [](const std::vector<int>& u, const std::vector<int>& v) { return u.size() > v.size(); });
      std::map<std::vector<int>, int> suffix_node;
      for (auto& s : order) suffix_node[s] = add_node(G, false);
      int succ = add_node(G, false);  // END or the node before the next gap
      auto node_for = [&](const std::vector<int>& suf) { return suf.empty() ? succ : suffix_node.at(suf); };
      std::set<std::tuple<int, int, int>> edge_set;
      for (auto& r : alts) {
        if (r.empty()) {
          edge_set.insert(std::make_tuple(pred, -1, succ));
          continue;
        }
        for (size_t t = 0; t < r.size(); ++t) {
          int from = (t == 0) ? pred : node_for(std::vector<int>(r.begin() + t, r.end()));
          int to = node_for(std::vector<int>(r.begin() + t + 1, r.end()));
          edge_set.insert(std::make_tuple(from, r[t], to));
        }
      }
      for (auto& e : edge_set) G.out[std::get<0>(e)].push_back({std::get<1>(e), std::get<2>(e)});
      cur = succ;
    }
    first = false;
    i = j;
  }
  G.accept = cur;
  return G;
}

// ------------------------------------------------------------------ Earley
// Alg. 3: worklist over items (node, production, dot, origin node).  The
// completion rule is applied in both orders (a new completed item advances
// the items already waiting at its origin; a new waiting item advances over
// completions already recorded), so the closure does not depend on the
// order in which the worklist is drained (nullable rules included).
struct EarleyStats {
  long long items = 0;
  std::vector<long long>* per_node_items = nullptr;     // optional census
  std::vector<std::set<int>>* per_node_origins = nullptr;
};

bool earley_valid(const Grammar& g, const Graph& G, bool early_exit, EarleyStats* st) {
  if (G.dead) return false;
  const int P = (int)g.rhs.size();
  auto key = [&](long long node, long long p, long long d, long long o) {
    return ((node * P + p) * 64 + d) * (long long)G.n_nodes + o;
  };
  std::unordered_set<long long> seen;
  struct Item {
    int node, p, d, o;
  };
  std::vector<Item> work;
  // waiting[(o, B)] -> items at node o waiting on B ; completed[(o,B)] -> end nodes
  std::unordered_map<long long, std::vector<Item>> waiting;
  std::unordered_map<long long, std::vector<int>> completed;
  std::unordered_map<long long, std::unordered_set<int>> completed_set;
  auto nb = [&](int o, int B) { return (long long)o * (g.T + g.V + 1) + B; };
  auto add = [&](int node, int p, int d, int o) {
    long long k = key(node, p, d, o);
    if (seen.insert(k).second) work.push_back({node, p, d, o});
  };
  add(G.start, g.aug, 0, G.start);
  while (!work.empty()) {
    Item it = work.back();
    work.pop_back();
    if (st) {
      st->items++;
      if (st->per_node_items) (*st->per_node_items)[it.node]++;
      if (st->per_node_origins) (*st->per_node_origins)[it.node].insert(it.o);
    }
    const std::vector<int>& r = g.rhs[it.p];
    // items move along epsilon edges unchanged
    for (auto& e : G.out[it.node])
      if (e.first < 0) add(e.second, it.p, it.d, it.o);
    if (it.d < (int)r.size()) {
      int X = r[it.d];
      if (X < g.T) {  // scan along matching terminal edges (and the gap loop)
        for (auto& e : G.out[it.node])
          if (e.first == X) add(e.second, it.p, it.d + 1, it.o);
        if (G.gap[it.node]) add(it.node, it.p, it.d + 1, it.o);
      } else {  // predict, and advance over completions already recorded
        waiting[nb(it.node, X)].push_back(it);
        for (int q : g.prods_of[X - g.T]) add(it.node, q, 0, it.node);
        auto c = completed.find(nb(it.node, X));
        if (c != completed.end()) {
          std::vector<int> ends = c->second;
          for (int j : ends) add(j, it.p, it.d + 1, it.o);
        }
      }
    } else {  // complete
      int B = g.lhs[it.p];
      if (it.p == g.aug) {
        if (it.node == G.accept && it.o == G.start && early_exit) return true;
        continue;
      }
      long long kb = nb(it.o, B + g.T);
      if (completed_set[kb].insert(it.node).second) {
        completed[kb].push_back(it.node);
        auto w = waiting.find(kb);
        if (w != waiting.end()) {
          std::vector<Item> ws = w->second;
          for (auto& wi : ws) add(it.node, wi.p, wi.d + 1, wi.o);
        }
      }
    }
  }
  return seen.count(key(G.accept, g.aug, 1, G.start)) > 0;
}

// ------------------------------------------------------------------ cover
// Regular cover F_G (Sec. 4.3, App. A.2, App. D.3): one network of states per
// grammar with its calls flattened.  States entry(A), exit(A) and (p, j) for
// every production p and dot j.  Every call site, recursive or not, goes to
// the one shared entry(B); exit(B) returns to every continuation of B.
struct Cover {
  int n = 0;
  std::vector<std::vector<std::pair<int, int>>> edges;  // (label, target), -1 = epsilon
  int start = 0, accept = 0;
};

// The cover is built from the reduced grammar (unproductive and unreachable
// nonterminals and the productions using them removed; L(G) is unchanged):
// a flattened network keeps return edges into every production that
// mentions a symbol, so useless productions would otherwise add paths.
std::vector<char> usable_productions(const Grammar& g) {
  int P = (int)g.rhs.size();
  std::vector<char> productive(g.V, 0);
  for (bool changed = true; changed;) {
    changed = false;
    for (int p = 0; p < P; ++p) {
      if (p == g.aug || productive[g.lhs[p]]) continue;
      bool all = true;
      for (int s : g.rhs[p])
        if (s >= g.T && !productive[s - g.T]) all = false;
      if (all) productive[g.lhs[p]] = 1, changed = true;
    }
  }
  auto ok = [&](int p) {
    if (!productive[g.lhs[p]]) return false;
    for (int s : g.rhs[p])
      if (s >= g.T && !productive[s - g.T]) return false;
    return true;
  };
  std::vector<char> reachable(g.V, 0);
  reachable[g.start] = 1;
  for (bool changed = true; changed;) {
    changed = false;
    for (int p = 0; p < P; ++p) {
      if (p == g.aug || !reachable[g.lhs[p]] || !ok(p)) continue;
      for (int s : g.rhs[p])
        if (s >= g.T && !reachable[s - g.T]) reachable[s - g.T] = 1, changed = true;
    }
  }
  std::vector<char> use(P, 0);
  for (int p = 0; p < P; ++p) use[p] = (p != g.aug) && reachable[g.lhs[p]] && ok(p);
  return use;
}

Cover build_cover(const Grammar& g) {
  Cover F;
  int V = g.V;
  std::vector<char> use = usable_productions(g);
  std::vector<int> base(g.rhs.size());
  int n = 2 * V;
  for (size_t p = 0; p < g.rhs.size(); ++p) {
    if ((int)p == g.aug) continue;
    base[p] = n;
    n += (int)g.rhs[p].size() + 1;
  }
  F.n = n;
  F.edges.assign(n, {});
  auto entry = [&](int A) { return A; };
  auto exitn = [&](int A) { return V + A; };
  for (size_t p = 0; p < g.rhs.size(); ++p) {
    if (!use[p]) continue;
    int A = g.lhs[p];
    const auto& r = g.rhs[p];
    F.edges[entry(A)].push_back({-1, base[p]});
    for (size_t j = 0; j < r.size(); ++j) {
      int X = r[j];
      if (X < g.T) {
        F.edges[base[p] + j].push_back({X, base[p] + (int)j + 1});
      } else {
        F.edges[base[p] + j].push_back({-1, entry(X - g.T)});
        F.edges[exitn(X - g.T)].push_back({-1, base[p] + (int)j + 1});
      }
    }
    F.edges[base[p] + r.size()].push_back({-1, exitn(A)});
  }
  F.start = entry(g.start);
  F.accept = exitn(g.start);
  return F;
}

void cover_eps_close(const Cover& F, std::vector<char>& s) {
  std::vector<int> stack;
  for (int i = 0; i < F.n; ++i)
    if (s[i]) stack.push_back(i);
  while (!stack.empty()) {
    int u = stack.back();
    stack.pop_back();
    for (auto& e : F.edges[u])
      if (e.first < 0 && !s[e.second]) {
        s[e.second] = 1;
        stack.push_back(e.second);
      }
  }
}

void cover_all_close(const Cover& F, std::vector<char>& s) {  // Sigma_lex* at a gap
  std::vector<int> stack;
  for (int i = 0; i < F.n; ++i)
    if (s[i]) stack.push_back(i);
  while (!stack.empty()) {
    int u = stack.back();
    stack.pop_back();
    for (auto& e : F.edges[u])
      if (!s[e.second]) {
        s[e.second] = 1;
        stack.push_back(e.second);
      }
  }
}

// L(F_G) cap L(A_x) != empty, by forward state-set simulation over the
// graph in node order (nodes are created in topological order).
bool cover_valid(const Grammar& g, const Cover& F, const Graph& G) {
  if (G.dead) return false;
  std::vector<std::vector<char>> S(G.n_nodes, std::vector<char>(F.n, 0));
  S[G.start][F.start] = 1;
  for (int u = 0; u < G.n_nodes; ++u) {
    cover_eps_close(F, S[u]);
    if (G.gap[u]) cover_all_close(F, S[u]);
    for (auto& e : G.out[u]) {
      int v = e.second;
      if (e.first < 0) {
        for (int i = 0; i < F.n; ++i)
          if (S[u][i]) S[v][i] = 1;
      } else {
        for (int i = 0; i < F.n; ++i)
          if (S[u][i])
            for (auto& fe : F.edges[i])
              if (fe.first == e.first) S[v][fe.second] = 1;
      }
    }
  }
  return S[G.accept][F.accept] != 0;
}

// ------------------------------------------------------------------ helpers
std::vector<int> apply_updates(const std::vector<int>& x, const std::vector<std::pair<int, int>>& upd) {
  std::vector<int> y = x;
  for (auto& u : upd) y[u.first] = u.second;  // (x (+) Delta)_j, Sec. 3
  return y;
}

bool exact_valid(const Grammar& g, const std::vector<int>& x, LexMemo& memo) {
  Graph G = build_graph(g, x, memo);
  return earley_valid(g, G, true, nullptr);
}

struct Cand {
  int slot;  // index into the proposed positions
  int pos, tok;
  float conf;
};

using CandList = std::vector<Cand>;

std::vector<std::pair<int, int>> as_updates(const CandList& c) {
  std::vector<std::pair<int, int>> u;
  for (auto& e : c) u.push_back({e.pos, e.tok});
  return u;
}

// the more confident half: the first ceil(|C|/2) of the confidence order
void split_halves(const CandList& c, CandList& L, CandList& R) {
  size_t h = (c.size() + 1) / 2;
  L.assign(c.begin(), c.begin() + h);
  R.assign(c.begin() + h, c.end());
}

struct Selector {
  const Grammar& g;
  const Cover& F;
  LexMemo memo;
  long long cover_checks = 0, exact_checks = 0;

  // Alg. 4, RelaxedSelect
  CandList relaxed(const std::vector<int>& x, const CandList& C) {
    if (C.size() <= 1) return {};
    std::vector<int> xc = apply_updates(x, as_updates(C));
    cover_checks++;
    Graph G = build_graph(g, xc, memo);
    if (cover_valid(g, F, G)) return C;
    CandList CL, CR;
    split_halves(C, CL, CR);
    CandList BL = relaxed(x, CL);
    CandList BR = relaxed(apply_updates(x, as_updates(BL)), CR);
    CandList out = BL;
    out.insert(out.end(), BR.begin(), BR.end());
    return out;
  }
  // Alg. 4, ExactShrink
  CandList shrink(const std::vector<int>& x, const CandList& B) {
    if (B.size() <= 1) return {};
    exact_checks++;
    if (exact_valid(g, apply_updates(x, as_updates(B)), memo)) return B;
    CandList BL, BR;
    split_halves(B, BL, BR);
    CandList BLp = shrink(x, BL);
    std::vector<int> xl = apply_updates(x, as_updates(BLp));
    CandList BRp = relaxed(xl, BR);
    CandList BRpp = shrink(xl, BRp);
    CandList out = BLp;
    out.insert(out.end(), BRpp.begin(), BRpp.end());
    return out;
  }
};

struct Oracle {
  Grammar g;
  Cover F;
  bool cover_built = false;
};

}  // namespace

// ====================================================================== C API
extern "C" {

void* orc_grammar_new(int T, const char* const* regex, const uint8_t* skip, int V, int start, int P,
                      const int* lhs, const int* rhs_off, const int* rhs, char* err, int errcap) {
  Oracle* O = new Oracle();
  Grammar& g = O->g;
  try {
    g.T = T;
    g.V = V;
    g.start = start;
    g.skip.assign(skip, skip + T);
    for (int t = 0; t < T; ++t) {
      RegexParser rp(g.nfa, regex[t]);
      Frag f = rp.parse_alt();
      if (rp.i != rp.s.size()) throw std::runtime_error("trailing regex input");
      g.nfa[f.accept].accept_term = t;
      g.term_start.push_back(f.start);
    }
    g.q0 = eclose(g, g.term_start);
    if (accepts(g, g.q0) >= 0) throw std::runtime_error("a terminal matches the empty string");
    // every lexer state reachable from q0 (the subset simulation's states);
    // all are live because every Thompson state lies on a path to an accept
    std::vector<std::vector<int>> todo{g.q0};
    g.state_id[g.q0] = 0;
    g.states.push_back(g.q0);
    while (!todo.empty()) {
      std::vector<int> q = todo.back();
      todo.pop_back();
      for (int c = 0; c < 256; ++c) {
        std::vector<int> n = step(g, q, c);
        if (n.empty() || g.state_id.count(n)) continue;
        g.state_id[n] = (int)g.states.size();
        g.states.push_back(n);
        todo.push_back(n);
      }
    }
    g.prods_of.assign(V, {});
    for (int p = 0; p < P; ++p) {
      g.lhs.push_back(lhs[p]);
      g.rhs.emplace_back(rhs + rhs_off[p], rhs + rhs_off[p + 1]);
      for (int s : g.rhs.back())
        if (s < 0 || s >= T + V || (s < T && skip[s])) throw std::runtime_error("bad rhs symbol");
      g.prods_of[lhs[p]].push_back(p);
    }
    g.aug = P;  // S' -> S  (S' is not a member of V; it is only ever completed)
    g.lhs.push_back(-1);
    g.rhs.push_back({T + start});
  } catch (std::exception& e) {
    if (err && errcap > 0) {
      strncpy(err, e.what(), errcap - 1);
      err[errcap - 1] = 0;
    }
    delete O;
    return nullptr;
  }
  return O;
}

void orc_grammar_free(void* h) { delete (Oracle*)h; }

int orc_num_lexer_states(void* h) { return (int)((Oracle*)h)->g.states.size(); }

void orc_set_vocab(void* h, int V, const int* off, const uint8_t* bytes) {
  Grammar& g = ((Oracle*)h)->g;
  g.vocab.clear();
  for (int t = 0; t < V; ++t) g.vocab.emplace_back((const char*)bytes + off[t], off[t + 1] - off[t]);
}

// Lex a byte string from lexer state `entry` (index into the live states,
// 0 = q0).  mode: 0 = the run only (pending lexeme left open), 1 = END
// flush, 2 = a gap follows.  Returns the run length, -1 if DEAD, -2 if cap
// is too small.  *pending receives the index of the pending state.
int orc_lex(void* h, int entry, const uint8_t* s, int len, int mode, int* out, int cap,
            int* pending) {
  Grammar& g = ((Oracle*)h)->g;
  std::vector<int> run, pend;
  if (!lex_run_mode(g, g.states[entry], std::string((const char*)s, len), mode, run, pend))
    return -1;
  if ((int)run.size() > cap) return -2;
  std::copy(run.begin(), run.end(), out);
  if (pending) *pending = g.state_id.count(pend) ? g.state_id.at(pend) : -1;
  return (int)run.size();
}

// Export the graph A_x.  Returns the number of edges (or -1 if cap too small);
// edges as (src, dst, label) triples, label -1 = epsilon.
int orc_graph(void* h, const int* x, int n, int* n_nodes, uint8_t* gap, int gap_cap, int* edges,
              int edge_cap, int* start, int* accept, int* dead) {
  Grammar& g = ((Oracle*)h)->g;
  LexMemo memo;
  Graph G = build_graph(g, std::vector<int>(x, x + n), memo);
  *n_nodes = G.n_nodes;
  *start = G.start;
  *accept = G.accept;
  *dead = G.dead;
  if (G.n_nodes > gap_cap) return -1;
  for (int u = 0; u < G.n_nodes; ++u) gap[u] = G.gap[u];
  int m = 0;
  for (int u = 0; u < G.n_nodes; ++u)
    for (auto& e : G.out[u]) {
      if (m >= edge_cap) return -1;
      edges[3 * m] = u;
      edges[3 * m + 1] = e.second;
      edges[3 * m + 2] = e.first;
      ++m;
    }
  return m;
}

// Completability of one partial output (token ids, -1 = MASK).
int orc_valid(void* h, const int* x, int n, long long* items) {
  Grammar& g = ((Oracle*)h)->g;
  EarleyStats st;
  LexMemo memo;
  Graph G = build_graph(g, std::vector<int>(x, x + n), memo);
  bool v = earley_valid(g, G, items == nullptr, items ? &st : nullptr);
  if (items) *items = st.items;
  return v ? 1 : 0;
}

// Chart census of the full (exhaustive) chart: items and distinct origins per
// node (a measurement aid).
int orc_chart_census(void* h, const int* x, int n, long long* items, int* origins, uint8_t* gap, int cap) {
  Grammar& g = ((Oracle*)h)->g;
  LexMemo memo;
  Graph G = build_graph(g, std::vector<int>(x, x + n), memo);
  if (G.n_nodes > cap) return -1;
  std::vector<long long> pi(G.n_nodes, 0);
  std::vector<std::set<int>> po(G.n_nodes);
  EarleyStats st;
  st.per_node_items = &pi;
  st.per_node_origins = &po;
  earley_valid(g, G, false, &st);
  for (int u = 0; u < G.n_nodes; ++u) {
    items[u] = pi[u];
    origins[u] = (int)po[u].size();
    gap[u] = G.gap[u];
  }
  return G.n_nodes;
}

// Is the terminal sequence the label of a path of x's partial-output graph,
// from its start node to its accept node (epsilon edges free, a gap node
// reading any terminal on its self-loop)?  The graph's language is C_x of
// Sec. 3 at the lexeme level, so with orc_accepts_terms this checks a witness
// completion (Sec. 4.4): a string of L(G) compatible with x.  Forward
// state-set simulation.
int orc_graph_accepts_terms(void* h, const int* x, int n, const int* terms, int len) {
  Grammar& g = ((Oracle*)h)->g;
  LexMemo memo;
  Graph G = build_graph(g, std::vector<int>(x, x + n), memo);
  if (G.dead) return 0;
  auto eps_close = [&](std::vector<char>& S) {
    std::vector<int> stack;
    for (int u = 0; u < G.n_nodes; ++u)
      if (S[u]) stack.push_back(u);
    while (!stack.empty()) {
      int u = stack.back();
      stack.pop_back();
      for (auto& e : G.out[u])
        if (e.first < 0 && !S[e.second]) {
          S[e.second] = 1;
          stack.push_back(e.second);
        }
    }
  };
  std::vector<char> S(G.n_nodes, 0);
  S[G.start] = 1;
  eps_close(S);
  for (int i = 0; i < len; ++i) {
    std::vector<char> N(G.n_nodes, 0);
    for (int u = 0; u < G.n_nodes; ++u) {
      if (!S[u]) continue;
      if (G.gap[u]) N[u] = 1;  // the gap's self-loop reads any terminal
      for (auto& e : G.out[u])
        if (e.first == terms[i]) N[e.second] = 1;
    }
    eps_close(N);
    S.swap(N);
  }
  return S[G.accept] ? 1 : 0;
}

// Earley acceptance of a plain terminal string (a graph that is one path).
int orc_accepts_terms(void* h, const int* terms, int len) {
  Grammar& g = ((Oracle*)h)->g;
  Graph G;
  int prev = add_node(G, false);
  G.start = prev;
  for (int i = 0; i < len; ++i) {
    int nx = add_node(G, false);
    G.out[prev].push_back({terms[i], nx});
    prev = nx;
  }
  G.accept = prev;
  return earley_valid(g, G, true, nullptr) ? 1 : 0;
}

static Cover& cover_of(Oracle* O) {
  if (!O->cover_built) {
    O->F = build_cover(O->g);
    O->cover_built = true;
  }
  return O->F;
}

int orc_cover_accepts_terms(void* h, const int* terms, int len) {
  Oracle* O = (Oracle*)h;
  Graph G;
  int prev = add_node(G, false);
  G.start = prev;
  for (int i = 0; i < len; ++i) {
    int nx = add_node(G, false);
    G.out[prev].push_back({terms[i], nx});
    prev = nx;
  }
  G.accept = prev;
  return cover_valid(O->g, cover_of(O), G) ? 1 : 0;
}

int orc_cover_valid(void* h, const int* x, int n) {
  Oracle* O = (Oracle*)h;
  LexMemo memo;
  Graph G = build_graph(O->g, std::vector<int>(x, x + n), memo);
  return cover_valid(O->g, cover_of(O), G) ? 1 : 0;
}

// valid[b][j][c] = Valid_G(x_b, {(pos[b][j], cand[b][j][c])}).  Returns 0,
// or -1 if a proposed position is not masked.  Checks are independent and
// are spread over nthreads threads (the CPU baseline's thread pool).
int orc_validate_batch(void* h, const int* x, int B, int n, const int* pos, int k, const int* cand,
                       int K, uint8_t* valid, int nthreads, long long* items_out) {
  Grammar& g = ((Oracle*)h)->g;
  for (int b = 0; b < B; ++b)
    for (int j = 0; j < k; ++j)
      if (pos[b * k + j] < 0 || pos[b * k + j] >= n || x[(long long)b * n + pos[b * k + j]] >= 0)
        return -1;
  long long total = (long long)B * k * K;
  std::atomic<long long> next(0);
  std::vector<long long> items(std::max(1, nthreads), 0);
  auto worker = [&](int w) {
    LexMemo memo;  // one cache per worker thread
    for (;;) {
      long long c = next.fetch_add(1);
      if (c >= total) break;
      int b = (int)(c / ((long long)k * K));
      int j = (int)((c / K) % k);
      std::vector<int> xs(x + (long long)b * n, x + (long long)(b + 1) * n);
      xs[pos[b * k + j]] = cand[c];
      Graph G = build_graph(g, xs, memo);
      EarleyStats st;
      valid[c] = earley_valid(g, G, items_out == nullptr, items_out ? &st : nullptr) ? 1 : 0;
      items[w] += st.items;
    }
  };
  if (nthreads <= 1) {
    worker(0);
  } else {
    std::vector<std::thread> th;
    for (int w = 0; w < nthreads; ++w) th.emplace_back(worker, w);
    for (auto& t : th) t.join();
  }
  if (items_out) {
    long long s = 0;
    for (long long v : items) s += v;
    *items_out = s;
  }
  return 0;
}

// Alg. 4 per sequence.  tok[b][j] is the candidate for proposed slot j (-1 =
// none) with confidence conf[b][j]; selected[b][j] = 1 for the committed
// batch.  Candidates are ordered by descending confidence, ties by
// ascending position.  Returns 0, -1 on a bad position, -2 on a NaN.
int orc_select(void* h, const int* x, int B, int n, const int* pos, int k, const int* tok,
               const float* conf, uint8_t* selected, long long* n_cover, long long* n_exact) {
  Oracle* O = (Oracle*)h;
  Grammar& g = O->g;
  Selector S{g, cover_of(O)};
  for (int b = 0; b < B; ++b) {
    CandList C;
    for (int j = 0; j < k; ++j) {
      selected[b * k + j] = 0;
      if (tok[b * k + j] < 0) continue;
      int p = pos[b * k + j];
      if (p < 0 || p >= n || x[(long long)b * n + p] >= 0) return -1;
      float c = conf[b * k + j];
      if (c != c) return -2;
      C.push_back({j, p, tok[b * k + j], c});
    }
    std::stable_sort(C.begin(), C.end(), [](const Cand& a, const Cand& c) {
      if (a.conf != c.conf) return a.conf > c.conf;
      return a.pos < c.pos;
    });
    std::vector<int> xs(x + (long long)b * n, x + (long long)(b + 1) * n);
    CandList Bsel = S.shrink(xs, S.relaxed(xs, C));
    for (auto& e : Bsel) selected[b * k + e.slot] = 1;
  }
  if (n_cover) *n_cover = S.cover_checks;
  if (n_exact) *n_exact = S.exact_checks;
  return 0;
}

// Sequential rejection fallback (Alg. 1, the loop after the selected batch
// B is committed): for each of the fill[b] = max(0, n_target[b] - |B|)
// remaining commits, take the highest-confidence candidate (over every
// proposed position and its K candidates) whose position is still masked and
// that was not rejected; while x (+) c fails the exact test of Sec. 3, reject
// it (its logit is suppressed) and take the next; commit the accepted one to
// x.  Readings: candidates are ordered by descending confidence, then
// ascending position, then ascending candidate index; positions committed
// before (by B or earlier in this loop) are not candidates; the loop stops
// early when no candidate is left.  x is updated in place; filled[b][j] =
// the token committed at slot j by this loop, else -1; *checks counts exact
// tests.  selected may be NULL (|B| = 0).  Returns -2 on a NaN confidence
// (nothing of that sequence is committed), -1 on a position out of range.
int orc_fallback(void* h, int* x, int B, int n, const int* pos, int k, const int* cand, const float* conf, int K,
                 const int* n_target, const uint8_t* selected, int* filled, long long* checks) {
  Oracle* O = (Oracle*)h;
  Grammar& g = O->g;
  LexMemo memo;
  long long nchk = 0;
  int ret = 0;
  for (int b = 0; b < B; ++b) {
    int* xb = x + (long long)b * n;
    for (int j = 0; j < k; ++j) filled[b * k + j] = -1;
    int nsel = 0;
    if (selected)
      for (int j = 0; j < k; ++j) nsel += selected[b * k + j] == 1;
    int fill = n_target[b] - nsel;
    struct Q {
      int j, c, p, t;
      float cf;
    };
    std::vector<Q> order;
    bool nan = false;
    for (int j = 0; j < k; ++j) {
      int p = pos[b * k + j];
      if (p < 0 || p >= n) return -1;
      for (int c = 0; c < K; ++c) {
        float cf = conf[((long long)b * k + j) * K + c];
        if (cf != cf) nan = true;
        order.push_back({j, c, p, cand[((long long)b * k + j) * K + c], cf});
      }
    }
    if (nan) {
      ret = -2;
      continue;
    }
    std::stable_sort(order.begin(), order.end(), [](const Q& a, const Q& q) {
      if (a.cf != q.cf) return a.cf > q.cf;
      if (a.p != q.p) return a.p < q.p;
      return a.c < q.c;
    });
    std::vector<char> rejected(order.size(), 0);
    for (int r = 0; r < fill; ++r) {
      bool committed = false;
      for (size_t q = 0; q < order.size() && !committed; ++q) {
        if (rejected[q] || xb[order[q].p] >= 0) continue;  // committed positions are not candidates
        std::vector<int> y(xb, xb + n);
        y[order[q].p] = order[q].t;
        ++nchk;
        if (order[q].t >= 0 && exact_valid(g, y, memo)) {
          xb[order[q].p] = order[q].t;
          filled[b * k + order[q].j] = order[q].t;
          committed = true;
        } else {
          rejected[q] = 1;
        }
      }
      if (!committed) break;  // every candidate rejected
    }
  }
  if (checks) *checks = nchk;
  return ret;
}

// Commit (Alg. 1): write the selected tokens into x.
void orc_commit(int* x, int B, int n, const int* pos, int k, const int* tok, const uint8_t* selected) {
  for (int b = 0; b < B; ++b)
    for (int j = 0; j < k; ++j)
      if (selected[b * k + j]) x[(long long)b * n + pos[b * k + j]] = tok[b * k + j];
}

}  // extern "C"

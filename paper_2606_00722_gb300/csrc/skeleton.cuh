// The graph walk shared by exact recognition (EarleyCols) and the cover
// group test (CoverCols): it enumerates the nodes of the partial-output graph
// of x (+) Delta in topological order, building them from the lex table, and
// asks the column type to combine, close and store each node.
#pragma once
#include "cover.cuh"
#include "walk.cuh"

namespace epic {

template <class Cols>
struct Walk {
  Cols& cols;
  const DevGrammar& g;
  const LexEntry* table;
  WalkScratch sc;
  WalkShared& sh;
  int vocab;
  const BlockRec* rec = nullptr;  // recording walks: positions' columns

  __device__ Walk(Cols& c, const DevGrammar& g_, const LexEntry* t, WalkScratch s, WalkShared& shared, int v)
      : cols(c), g(g_), table(t), sc(s), sh(shared), vocab(v) {}

  __device__ void label_set(const uint32_t* lbl8) {
    if (Cols::kRecord && threadIdx.x < 8) sh.lbl8[threadIdx.x] = lbl8[threadIdx.x];
    for (int w = threadIdx.x; w < g.W; w += blockDim.x) {
      uint32_t acc = 0;
      for (int lw = 0; lw < 8; ++lw) {
        uint32_t m = lbl8[lw];
        while (m) {
          int b = __ffs(m) - 1;
          m &= m - 1;
          int a = (lw << 5) + b;
          if (a < g.T) acc |= g.exp_term[(size_t)a * g.W + w];
        }
      }
      sh.lbl[w] = acc;
    }
    __syncthreads();
  }
  __device__ void label_one(int a) {
    if (Cols::kRecord && threadIdx.x < 8) sh.lbl8[threadIdx.x] = (threadIdx.x == (a >> 5)) ? (1u << (a & 31)) : 0u;
    for (int w = threadIdx.x; w < g.W; w += blockDim.x) sh.lbl[w] = g.exp_term[(size_t)a * g.W + w];
    __syncthreads();
  }

  __device__ static int token_at(const int32_t* x, const Subst& s, int i) {
    for (int j = 0; j < s.n; ++j)
      if (s.pos[j] == i) return s.tok[j];
    return x[i];
  }

  // Arrival of group gi into its end node: (source column, label set), the
  // label set all zero for an epsilon edge.
  __device__ int arrival_src(int gi) const { return sc.g_len[gi] >= 2 ? sc.g_last[gi] : sc.g_src[gi]; }
  __device__ uint32_t arrival_lbl(int gi, int w) const {
    const int len = sc.g_len[gi];
    if (len == 0) return 0u;
    if (len == 1) return sc.g_lbl[gi * 8 + w];
    const int a = sc.g_tail[gi * 16 + len - 2];
    return (w == (a >> 5)) ? (1u << (a & 31)) : 0u;
  }
  // Do end states e1 and e2 receive the same arrivals?  (One thread.)
  __device__ bool same_arrivals(int e1, int e2, int ng) const {
    int n1 = 0, n2 = 0;
    for (int gi = 0; gi < ng; ++gi) {
      n1 += sc.g_end[gi] == e1;
      n2 += sc.g_end[gi] == e2;
    }
    if (n1 != n2) return false;
    for (int gi = 0; gi < ng; ++gi) {
      if (sc.g_end[gi] != e1) continue;
      bool found = false;
      for (int gj = 0; gj < ng && !found; ++gj) {
        if (sc.g_end[gj] != e2 || arrival_src(gj) != arrival_src(gi)) continue;
        bool same = (sc.g_len[gi] == 0) == (sc.g_len[gj] == 0);
        for (int w = 0; w < 8; ++w) same &= arrival_lbl(gi, w) == arrival_lbl(gj, w);
        found = same;
      }
      if (!found) return false;
    }
    return true;
  }

  // One token of a span: frontier (f_q lexer state, f_c column)[0..nf) ->
  // new frontier.  Lexings from the same column with the same end state and
  // the same terminals after the first share one path whose first edge
  // carries all their first terminals.  Returns false on overflow.
  __device__ bool span_step(int tok) {
    int nf = sh.nf;
    if (g.lazy.stats && threadIdx.x == 0) atomicAdd(&g.lazy.stats[0], (unsigned long long)nf);
    for (int f = threadIdx.x; f < nf; f += blockDim.x) {
      LexEntry e = lex_at(g, table, tok, sc.f_q[f]);
      int src = sc.f_c[f];
      int leader = -1;
      if (e.end != 0xFFFF) {
        leader = f;
        for (int h = 0; h < f; ++h) {
          if (sc.f_c[h] != src) continue;
          LexEntry e2 = lex_at(g, table, tok, sc.f_q[h]);
          if (e2.end != e.end || e2.len != e.len) continue;
          bool same = true;
          for (int t = 1; t < e.len; ++t) same &= e.term[t] == e2.term[t];
          if (same) {
            leader = h;
            break;
          }
        }
      }
      sc.key_q[f] = leader;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int ng = 0;
      for (int f = 0; f < nf; ++f) {
        if (sc.key_q[f] != f) continue;
        LexEntry e = lex_at(g, table, tok, sc.f_q[f]);
        sc.g_src[ng] = sc.f_c[f];
        sc.g_end[ng] = e.end;
        sc.g_len[ng] = e.len;
        for (int t = 0; t < 16; ++t) sc.g_tail[ng * 16 + t] = (t + 1 < e.len) ? e.term[t + 1] : 0;
        for (int w = 0; w < 8; ++w) sc.g_lbl[ng * 8 + w] = 0;
        sc.key_q[f] = -2 - ng;
        ++ng;
      }
      for (int f = 0; f < nf; ++f) {
        int k = sc.key_q[f];
        if (k == -1) continue;
        int gid = (k <= -2) ? (-2 - k) : (-2 - sc.key_q[k]);
        LexEntry e = lex_at(g, table, tok, sc.f_q[f]);
        if (e.len > 0) sc.g_lbl[gid * 8 + (e.term[0] >> 5)] |= 1u << (e.term[0] & 31);
      }
      sh.ng = ng;
    }
    __syncthreads();
    int ng = sh.ng;
    // the run up to its last terminal (intermediate nodes); groups with the
    // same source, first-terminal set and terminals before the last one
    // spell the same paths up to it, so they share one chain of nodes
    for (int gi = 0; gi < ng; ++gi) {
      int len = sc.g_len[gi];
      int cur = sc.g_src[gi];
      if (len >= 2) {
        if (threadIdx.x == 0) {
          int share = -1;
          for (int gj = 0; gj < gi && share < 0; ++gj) {
            if (sc.g_len[gj] != len || sc.g_src[gj] != cur) continue;
            bool same = true;
            for (int w = 0; w < 8; ++w) same &= sc.g_lbl[gj * 8 + w] == sc.g_lbl[gi * 8 + w];
            for (int t = 0; t + 2 < len; ++t) same &= sc.g_tail[gj * 16 + t] == sc.g_tail[gi * 16 + t];
            if (same) share = gj;
          }
          sh.scratch_i[0] = share;
        }
        __syncthreads();
        const int share = sh.scratch_i[0];
        __syncthreads();
        if (share >= 0) {
          if (threadIdx.x == 0) sc.g_last[gi] = sc.g_last[share];
          __syncthreads();
          continue;
        }
      }
      for (int t = 0; t + 1 < len; ++t) {
        int c = cols.open_column();
        __syncthreads();
        if (c < 0) return false;
        if (t == 0)
          label_set(sc.g_lbl + gi * 8);
        else
          label_one(sc.g_tail[gi * 16 + t - 1]);
        cols.arrive_labels(cur, false);
        cols.close_column(c, false);
        cols.finish_column(c);
        if (sh.status != kWalkOk) return false;
        cur = c;
      }
      if (threadIdx.x == 0) sc.g_last[gi] = cur;
      __syncthreads();
    }
    // one node per distinct end state, ascending
    if (threadIdx.x == 0) {
      int nt = 0;
      for (int gi = 0; gi < ng; ++gi) {
        int e = sc.g_end[gi];
        bool seen = false;
        for (int j = 0; j < nt; ++j) seen |= sc.f_q[j] == e;
        if (!seen) sc.f_q[nt++] = e;
      }
      for (int i = 1; i < nt; ++i) {
        int v = sc.f_q[i], j = i - 1;
        while (j >= 0 && sc.f_q[j] > v) {
          sc.f_q[j + 1] = sc.f_q[j];
          --j;
        }
        sc.f_q[j + 1] = v;
      }
      sh.nt = nt;
    }
    __syncthreads();
    int nt = sh.nt;
    // end nodes with the same arrivals (sources and labels) have the same
    // incoming paths: one column serves all their lexer states.  Each end's
    // arrivals are hashed (sh.list) and counted (sh.prefix, free until the
    // nodes are built); the smallest equal end is its representative.
    for (int ti = threadIdx.x; ti < nt; ti += blockDim.x) {
      const int e = sc.f_q[ti];
      uint32_t h = 0;
      int cnt = 0;
      for (int gi = 0; gi < ng; ++gi) {
        if (sc.g_end[gi] != e) continue;
        uint32_t x = (uint32_t)arrival_src(gi) * 0x9E3779B1u + (sc.g_len[gi] == 0 ? 0x85EBCA6Bu : 0u);
        for (int w = 0; w < 8; ++w) x = (x ^ arrival_lbl(gi, w)) * 0xC2B2AE35u + (uint32_t)w;
        h += x ^ (x >> 16);
        ++cnt;
      }
      sh.list[ti] = (int32_t)h;
      sh.prefix[ti] = cnt;
    }
    __syncthreads();
    for (int ti = threadIdx.x; ti < nt; ti += blockDim.x) {
      int rep = ti;
      for (int tj = 0; tj < ti; ++tj)
        if (sh.list[tj] == sh.list[ti] && sh.prefix[tj] == sh.prefix[ti] &&
            same_arrivals(sc.f_q[ti], sc.f_q[tj], ng)) {
          rep = tj;
          break;
        }
      sc.key_q[ti] = rep;
    }
    __syncthreads();
    for (int ti = 0; ti < nt; ++ti) {
      if (sc.key_q[ti] != ti) continue;
      int e = sc.f_q[ti];
      int c = cols.open_column();
      __syncthreads();
      if (c < 0) return false;
      for (int gi = 0; gi < ng; ++gi) {
        if (sc.g_end[gi] != e) continue;
        int len = sc.g_len[gi];
        if (len == 0) {
          cols.arrive_labels(sc.g_src[gi], true);
        } else if (len == 1) {
          label_set(sc.g_lbl + gi * 8);
          cols.arrive_labels(sc.g_src[gi], false);
        } else {
          label_one(sc.g_tail[gi * 16 + len - 2]);
          cols.arrive_labels(sc.g_last[gi], false);
        }
      }
      cols.close_column(c, false);
      cols.finish_column(c);
      if (sh.status != kWalkOk) return false;
      if (threadIdx.x == 0) sc.f_c[ti] = c;
      __syncthreads();
    }
    if (threadIdx.x == 0) {
      for (int ti = 0; ti < nt; ++ti)
        if (sc.key_q[ti] != ti) sc.f_c[ti] = sc.f_c[sc.key_q[ti]];
      int k = 0;
      for (int ti = 0; ti < nt; ++ti)
        if (!cols.column_empty(sc.f_c[ti])) {
          sc.f_q[k] = sc.f_q[ti];
          sc.f_c[k] = sc.f_c[ti];
          ++k;
        }
      sh.nf = k;
    }
    __syncthreads();
    return true;
  }

  // Walk x (+) s.  Returns 1 (accept item at the accept node), 0, -1 on a
  // capacity overflow, -2 on bad input (unmasked position, bad token id).
  __device__ int run(const int32_t* x, int n, Subst s) {
    cols.reset();
    if (threadIdx.x == 0) {
      for (int j = 0; j < s.n; ++j) {
        int p = s.pos[j];
        if (p < 0 || p >= n || x[p] >= 0 || s.tok[j] < 0 || s.tok[j] >= vocab) sh.status = kWalkBadInput;
      }
    }
    __syncthreads();
    if (sh.status != kWalkOk) return -2;
    int r = run_inner(x, n, s);
    if (r < 0) cols.cleanup();
    return r;
  }

  __device__ int seed_column(bool gap) {
    int c = cols.open_column();
    __syncthreads();
    if (c < 0) return -1;
    if (threadIdx.x == 0) sh.start_col = c;
    __syncthreads();
    cols.seed(c);
    return c;
  }

  // positions [lo, hi) of a recording walk -> column c
  __device__ void rec_range(int32_t* arr, int lo, int hi, int c) {
    for (int p = lo + threadIdx.x; p < hi; p += blockDim.x) arr[p] = c;
  }

  __device__ int run_inner(const int32_t* x, int n, Subst s) {
    if (n == 0) {
      int c = seed_column(false);
      if (c < 0) return -1;
      cols.close_column(c, false);
      cols.finish_column(c);
      if (sh.status != kWalkOk) return -1;
      if (threadIdx.x == 0) sh.accept_col = c;
      return cols.column_has_accept(c, c) ? 1 : 0;
    }
    int i = 0;
    bool first = true;
    int prev_gap = -1;
    int span_lo = -1, span_hi = -1;  // the last span (recording walks)
    while (i < n) {
      int t0 = token_at(x, s, i);
      int j = i;
      if (t0 < 0) {
        while (j < n && token_at(x, s, j) < 0) ++j;
        int c;
        if (first) {
          c = seed_column(true);
          if (c < 0) return -1;
        } else {
          c = cols.open_column();
          __syncthreads();
          if (c < 0) return -1;
          // the span before the gap: a pending lexeme that some byte can
          // extend stays open (the gap absorbs its terminal); one that no
          // byte can extend has ended and emits its terminal
          int nf = sh.nf;
          for (int f = 0; f < nf; ++f) {
            int q = sc.f_q[f];
            int a = g.dfa_accept[q];
            if (q == 0 || g.dfa_ext[q] || (a >= 0 && g.skip[a])) {
              cols.arrive_labels(sc.f_c[f], true);
            } else if (a >= 0) {
              label_one(a);
              cols.arrive_labels(sc.f_c[f], false);
            }
          }
        }
        cols.close_column(c, true);
        cols.finish_column(c);
        if (sh.status != kWalkOk) return -1;
        if (Cols::kRecord) {
          rec_range(rec->gap_col, i, j, c);
          if (span_lo >= 0) rec_range(rec->post_col, span_lo, span_hi, c);
        }
        prev_gap = c;
        if (cols.column_empty(c)) return 0;
      } else {
        while (j < n && token_at(x, s, j) >= 0) ++j;
        if (first) {
          int c = seed_column(false);
          if (c < 0) return -1;
          cols.close_column(c, false);
          cols.finish_column(c);
          if (sh.status != kWalkOk) return -1;
          if (threadIdx.x == 0) {
            sc.f_q[0] = 0;
            sc.f_c[0] = c;
            sh.nf = 1;
          }
          if (Cols::kRecord) rec_range(rec->pre_col, i, j, c);
        } else {
          if (Cols::kRecord) rec_range(rec->pre_col, i, j, prev_gap);
          for (int q = threadIdx.x; q < g.Q; q += blockDim.x) {
            sc.f_q[q] = q;
            sc.f_c[q] = prev_gap;
          }
          if (threadIdx.x == 0) sh.nf = g.Q;
        }
        __syncthreads();
        span_lo = i;
        span_hi = j;
        for (int p = i; p < j; ++p) {
          if (sh.nf == 0) break;
          int tok = token_at(x, s, p);
          if (tok < 0 || tok >= vocab) return -2;
          if (!span_step(tok)) return -1;
        }
        if (sh.nf == 0) return 0;  // no lexing of this span survives
        if (j == n) {              // END: flush the pending lexeme
          int c = cols.open_column();
          __syncthreads();
          if (c < 0) return -1;
          int nf = sh.nf;
          for (int f = 0; f < nf; ++f) {
            int q = sc.f_q[f];
            int a = g.dfa_accept[q];
            if (q == 0 || (a >= 0 && g.skip[a])) {
              cols.arrive_labels(sc.f_c[f], true);
            } else if (a >= 0) {
              label_one(a);
              cols.arrive_labels(sc.f_c[f], false);
            }
          }
          cols.close_column(c, false);
          cols.finish_column(c);
          if (sh.status != kWalkOk) return -1;
          if (Cols::kRecord) rec_range(rec->post_col, i, j, c);
          if (threadIdx.x == 0) sh.accept_col = c;
          return cols.column_has_accept(c, sh.start_col) ? 1 : 0;
        }
      }
      first = false;
      i = j;
    }
    if (threadIdx.x == 0) sh.accept_col = prev_gap;
    return cols.column_has_accept(prev_gap, sh.start_col) ? 1 : 0;
  }
};

}  // namespace epic

"""EPIC validity oracle -- test infrastructure only.

A plain CPU implementation (``epic_oracle.cpp``) of what the hot path
computes, written from the paper: the completability predicate of Sec. 3,
the partial-output graph of Alg. 2, the Earley-style graph parser of Alg. 3,
the flattened regular cover of Sec. 4.3 / App. A.2, Alg. 4's relaxed
subset selection with exact shrink, and Alg. 1's sequential rejection
fallback.  It shares no code with the CUDA path.

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg and reference arm may import this module.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, 'epic_oracle.cpp')
_OUT = os.path.join(_HERE, '_build', 'libepic_oracle.so')
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with the host C++ compiler (no CUDA involved)."""
    os.makedirs(os.path.dirname(_OUT), exist_ok=True)
    if force or not os.path.exists(_OUT) or os.path.getmtime(_OUT) < os.path.getmtime(_SRC):
        tmp = _OUT + '.tmp%d' % os.getpid()
        subprocess.check_call(['g++', '-O2', '-std=c++17', '-shared', '-fPIC', '-pthread',
                               _SRC, '-o', tmp])
        os.replace(tmp, _OUT)
    return _OUT


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = C.CDLL(build())
            P = C.POINTER
            i32p, u8p, f32p, i64p = P(C.c_int32), P(C.c_uint8), P(C.c_float), P(C.c_longlong)
            lib.orc_grammar_new.restype = C.c_void_p
            lib.orc_grammar_new.argtypes = [C.c_int, P(C.c_char_p), u8p, C.c_int, C.c_int, C.c_int,
                                            i32p, i32p, i32p, C.c_char_p, C.c_int]
            lib.orc_grammar_free.argtypes = [C.c_void_p]
            lib.orc_num_lexer_states.argtypes = [C.c_void_p]
            lib.orc_set_vocab.argtypes = [C.c_void_p, C.c_int, i32p, u8p]
            lib.orc_lex.argtypes = [C.c_void_p, C.c_int, u8p, C.c_int, C.c_int, i32p, C.c_int, i32p]
            lib.orc_graph.argtypes = [C.c_void_p, i32p, C.c_int, i32p, u8p, C.c_int, i32p, C.c_int,
                                      i32p, i32p, i32p]
            lib.orc_valid.argtypes = [C.c_void_p, i32p, C.c_int, i64p]
            lib.orc_chart_census.argtypes = [C.c_void_p, i32p, C.c_int, i64p, i32p, u8p, C.c_int]
            lib.orc_accepts_terms.argtypes = [C.c_void_p, i32p, C.c_int]
            lib.orc_graph_accepts_terms.argtypes = [C.c_void_p, i32p, C.c_int, i32p, C.c_int]
            lib.orc_cover_accepts_terms.argtypes = [C.c_void_p, i32p, C.c_int]
            lib.orc_cover_valid.argtypes = [C.c_void_p, i32p, C.c_int]
            lib.orc_validate_batch.argtypes = [C.c_void_p, i32p, C.c_int, C.c_int, i32p, C.c_int,
                                               i32p, C.c_int, u8p, C.c_int, i64p]
            lib.orc_select.argtypes = [C.c_void_p, i32p, C.c_int, C.c_int, i32p, C.c_int, i32p,
                                       f32p, u8p, i64p, i64p]
            lib.orc_commit.argtypes = [i32p, C.c_int, C.c_int, i32p, C.c_int, i32p, u8p]
            lib.orc_fallback.argtypes = [C.c_void_p, i32p, C.c_int, C.c_int, i32p, C.c_int, i32p, f32p,
                                         C.c_int, i32p, u8p, i32p, i64p]
            _lib = lib
    return _lib


def _p(a, ct):
    return a.ctypes.data_as(C.POINTER(ct))


class Oracle:
    """Oracle bound to one grammar (and optionally a vocabulary)."""

    def __init__(self, grammar, vocab=None):
        lib = _load()
        self._lib = lib
        self.g = grammar
        T = grammar.T
        regs = (C.c_char_p * T)(*[t.regex.encode('latin-1') for t in grammar.terminals])
        skip = np.array([1 if t.skip else 0 for t in grammar.terminals], np.uint8)
        lhs, off, rhs = grammar.rhs_flat()
        rhs = rhs if rhs.size else np.zeros(1, np.int32)
        err = C.create_string_buffer(256)
        h = lib.orc_grammar_new(T, regs, _p(skip, C.c_uint8), grammar.V, grammar.start,
                                len(grammar.productions), _p(lhs, C.c_int32), _p(off, C.c_int32),
                                _p(rhs, C.c_int32), err, 256)
        if not h:
            raise ValueError('oracle rejected grammar: ' + err.value.decode())
        self.h = h
        self._keep = (regs, skip, lhs, off, rhs)
        if vocab is not None:
            self.set_vocab(vocab)

    def __del__(self):
        h = getattr(self, 'h', None)
        if h:
            self._lib.orc_grammar_free(h)
            self.h = None

    @property
    def n_lexer_states(self):
        return self._lib.orc_num_lexer_states(self.h)

    def set_vocab(self, vocab):
        lens = np.array([len(t) for t in vocab], np.int64)
        off = np.zeros(len(vocab) + 1, np.int32)
        off[1:] = np.cumsum(lens)
        data = np.frombuffer(b''.join(vocab) or b'\0', np.uint8).copy()
        self._lib.orc_set_vocab(self.h, len(vocab), _p(off, C.c_int32), _p(data, C.c_uint8))
        self.vocab = list(vocab)

    def lex(self, text: bytes, entry: int = 0, flush_end: bool = True, run_only: bool = False):
        """Greedy lexing of text from live lexer state `entry` (0 = initial):
        with the END flush, or as a span before a gap, or (run_only) with the
        pending lexeme left open.  Returns (run of terminal ids, pending
        state index) or None if DEAD."""
        buf = np.frombuffer(text or b'\0', np.uint8).copy()
        out = np.zeros(len(text) + 2, np.int32)
        pend = C.c_int32(-1)
        mode = 0 if run_only else (1 if flush_end else 2)
        r = self._lib.orc_lex(self.h, entry, _p(buf, C.c_uint8), len(text), mode,
                              _p(out, C.c_int32), len(out), C.byref(pend))
        if r == -1:
            return None
        return [int(v) for v in out[:r]], pend.value

    def graph(self, x):
        """The partial-output graph: (n_nodes, gap flags, edges[(u, v, label)],
        start, accept, dead).  label -1 is an epsilon edge."""
        x = np.ascontiguousarray(x, np.int32)
        cap_n, cap_e = 1 << 16, 1 << 18
        nn, st, ac, dd = C.c_int32(), C.c_int32(), C.c_int32(), C.c_int32()
        gap = np.zeros(cap_n, np.uint8)
        edges = np.zeros(3 * cap_e, np.int32)
        m = self._lib.orc_graph(self.h, _p(x, C.c_int32), len(x), C.byref(nn), _p(gap, C.c_uint8),
                                cap_n, _p(edges, C.c_int32), cap_e, C.byref(st), C.byref(ac),
                                C.byref(dd))
        if m < 0:
            raise RuntimeError('graph too large')
        e = edges[:3 * m].reshape(m, 3)
        return nn.value, gap[:nn.value].copy(), [tuple(int(v) for v in r) for r in e], \
            st.value, ac.value, bool(dd.value)

    def valid(self, x, count_items: bool = False):
        x = np.ascontiguousarray(x, np.int32)
        if count_items:
            it = C.c_longlong(0)
            v = self._lib.orc_valid(self.h, _p(x, C.c_int32), len(x), C.byref(it))
            return bool(v), it.value
        return bool(self._lib.orc_valid(self.h, _p(x, C.c_int32), len(x), None))

    def chart_census(self, x):
        """Per graph node: (items, distinct origins, is-gap) of the full chart."""
        x = np.ascontiguousarray(x, np.int32)
        cap = 1 << 16
        it = np.zeros(cap, np.int64)
        org = np.zeros(cap, np.int32)
        gap = np.zeros(cap, np.uint8)
        m = self._lib.orc_chart_census(self.h, _p(x, C.c_int32), len(x), _p(it, C.c_longlong),
                                       _p(org, C.c_int32), _p(gap, C.c_uint8), cap)
        return it[:m].copy(), org[:m].copy(), gap[:m].copy()

    def accepts_terms(self, terms):
        t = np.ascontiguousarray(terms if len(terms) else [0], np.int32)
        return bool(self._lib.orc_accepts_terms(self.h, _p(t, C.c_int32), len(terms)))

    def graph_accepts_terms(self, x, terms):
        """Is the terminal sequence a path label of x's partial-output graph
        (a lexeme sequence compatible with x, gaps reading anything)?"""
        x = np.ascontiguousarray(x, np.int32)
        t = np.ascontiguousarray(terms if len(terms) else [0], np.int32)
        return bool(self._lib.orc_graph_accepts_terms(self.h, _p(x, C.c_int32), len(x), _p(t, C.c_int32),
                                                       len(terms)))

    def cover_accepts_terms(self, terms):
        t = np.ascontiguousarray(terms if len(terms) else [0], np.int32)
        return bool(self._lib.orc_cover_accepts_terms(self.h, _p(t, C.c_int32), len(terms)))

    def cover_valid(self, x):
        x = np.ascontiguousarray(x, np.int32)
        return bool(self._lib.orc_cover_valid(self.h, _p(x, C.c_int32), len(x)))

    def validate_batch(self, x, pos, cand, nthreads: int = 1, count_items: bool = False):
        x = np.ascontiguousarray(x, np.int32)
        pos = np.ascontiguousarray(pos, np.int32)
        cand = np.ascontiguousarray(cand, np.int32)
        B, n = x.shape
        k = pos.shape[1]
        K = cand.shape[2]
        valid = np.zeros((B, k, K), np.uint8)
        it = C.c_longlong(0)
        r = self._lib.orc_validate_batch(self.h, _p(x, C.c_int32), B, n, _p(pos, C.c_int32), k,
                                         _p(cand, C.c_int32), K, _p(valid, C.c_uint8), nthreads,
                                         C.byref(it) if count_items else None)
        if r != 0:
            raise ValueError('a proposed position is not masked')
        return (valid, it.value) if count_items else valid

    def select(self, x, pos, tok, conf):
        x = np.ascontiguousarray(x, np.int32)
        pos = np.ascontiguousarray(pos, np.int32)
        tok = np.ascontiguousarray(tok, np.int32)
        conf = np.ascontiguousarray(conf, np.float32)
        B, n = x.shape
        k = pos.shape[1]
        sel = np.zeros((B, k), np.uint8)
        nc, ne = C.c_longlong(0), C.c_longlong(0)
        r = self._lib.orc_select(self.h, _p(x, C.c_int32), B, n, _p(pos, C.c_int32), k,
                                 _p(tok, C.c_int32), _p(conf, C.c_float), _p(sel, C.c_uint8),
                                 C.byref(nc), C.byref(ne))
        if r == -1:
            raise ValueError('a proposed position is not masked')
        if r == -2:
            raise ValueError('NaN confidence')
        self.last_select_counts = (nc.value, ne.value)
        return sel

    def fallback(self, x, pos, cand, conf, n_target, selected=None):
        """Alg. 1's sequential rejection fallback after the selected batch
        was committed (x already holds it): returns (x updated, filled [B][k]
        token committed at each slot by the fallback or -1, exact checks)."""
        x = np.array(x, np.int32, copy=True)
        pos = np.ascontiguousarray(pos, np.int32)
        cand = np.ascontiguousarray(cand, np.int32)
        conf = np.ascontiguousarray(conf, np.float32)
        n_target = np.ascontiguousarray(n_target, np.int32)
        B, n = x.shape
        k = pos.shape[1]
        K = cand.shape[2]
        filled = np.full((B, k), -1, np.int32)
        sel = None if selected is None else np.ascontiguousarray(selected, np.uint8)
        nchk = C.c_longlong(0)
        r = self._lib.orc_fallback(self.h, _p(x, C.c_int32), B, n, _p(pos, C.c_int32), k, _p(cand, C.c_int32),
                                   _p(conf, C.c_float), K, _p(n_target, C.c_int32),
                                   None if sel is None else _p(sel, C.c_uint8), _p(filled, C.c_int32),
                                   C.byref(nchk))
        if r == -1:
            raise ValueError('a proposed position is out of range')
        if r == -2:
            raise ValueError('NaN confidence')
        return x, filled, nchk.value

    @staticmethod
    def commit(x, pos, tok, selected):
        x = np.array(x, np.int32, copy=True)
        pos = np.ascontiguousarray(pos, np.int32)
        tok = np.ascontiguousarray(tok, np.int32)
        selected = np.ascontiguousarray(selected, np.uint8)
        B, n = x.shape
        _load().orc_commit(_p(x, C.c_int32), B, n, _p(pos, C.c_int32), pos.shape[1],
                           _p(tok, C.c_int32), _p(selected, C.c_uint8))
        return x


def pick_candidates(valid, cand, conf):
    """Per proposed position, the highest-confidence candidate whose valid bit
    is 1 (ties: lowest candidate index); (-1, 0) when none is valid."""
    B, k, K = cand.shape
    tok = np.full((B, k), -1, np.int32)
    cf = np.zeros((B, k), np.float32)
    for b in range(B):
        for j in range(k):
            best = -1
            for c in range(K):
                if valid[b, j, c] == 1 and (best < 0 or conf[b, j, c] > conf[b, j, best]):
                    best = c
            if best >= 0:
                tok[b, j] = cand[b, j, best]
                cf[b, j] = conf[b, j, best]
    return tok, cf

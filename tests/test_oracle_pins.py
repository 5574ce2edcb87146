"""Pins of the CPU oracle against facts that do not come from the oracle.

The paper has no printed worked example, so the oracle is pinned by
(i) hand-derived lexing cases, (ii) an independent greedy lexer built on the
`regex` module's partial matching, (iii) exhaustive language enumeration of
tiny grammars (textbook membership), (iv) an independent Bar-Hillel fixpoint
over the same partial-output graph (the intersection formulation of prior
work, Sec. 4.2 / App. A.2), (v) one-sided brute force over mask fillings,
(vi) the special cases that reduce to membership / non-emptiness / viable
prefixes, (vii) monotonicity (App. D), and (viii) for the regular cover,
L(G) subset L(F_G) and exactness on a non-recursive grammar (App. D.3).
"""
import itertools
import os

import numpy as np
import pytest

import oracle
from synth import grammars as G
from synth import make_workload, sample_derivation, render

HERE = os.path.dirname(os.path.abspath(__file__))


# ------------------------------------------------------------------ grammars
def expr():
    return G.expr_grammar()


def tiny_paren():
    """S -> ( S ) S | a ; plus an unused-in-L terminal b."""
    b = G._Builder('paren')
    b.lit('(')
    b.lit(')')
    b.lit('a')
    b.lit('b')
    b.term('WS', '[ ]+', ('ws',), skip=True)
    b.rule('S', '( S ) S', 'a')
    return b.build('S', '()ab ')


def tiny_nonrec():
    """Non-recursive grammar where every nonterminal occurs at most once on
    all right-hand sides: its flattened cover is exact."""
    b = G._Builder('nonrec')
    for c in 'abcde':
        b.lit(c)
    b.rule('S', 'A B', 'c')
    b.rule('A', 'a', 'a d')
    b.rule('B', 'b', 'e')
    return b.build('S', 'abcde', has_ws=False)


def tiny_eps():
    """Grammar with epsilon productions and nullable chains."""
    b = G._Builder('eps')
    for c in 'xyz':
        b.lit(c)
    b.rule('S', 'A S B', 'z')
    b.rule('A', 'x', [])
    b.rule('B', 'y', 'A')
    return b.build('S', 'xyz', has_ws=False)


def words_grammar():
    """Identifier/keyword/number lexing with a one-byte-lookahead dead end."""
    b = G._Builder('words')
    b.lit('if', 'IF')
    b.lit('<<=', 'SHLEQ')
    b.lit('<', 'LT')
    b.term('ID', '[a-z]+', ('word', 'ab', 'ab', 1, 3))
    b.term('NUM', '[0-9]+(\\.[0-9]+)?', ('digits', 1, 2))
    b.term('WS', '[ ]+', ('ws',), skip=True)
    b.rule('S', 'S X', 'X')
    b.rule('X', 'IF', 'SHLEQ', 'LT', 'ID', 'NUM')
    return b.build('S', 'abfi<=0123. ')


# ------------------------------------------------------------------ helpers
def language(g, maxlen):
    """All terminal strings of length <= maxlen derivable from the start symbol
    (leftmost expansion of sentential forms; exact for grammars whose
    nonterminals all derive a non-empty string or epsilon finitely)."""
    T = g.T
    out = set()
    seen = set()
    frontier = [(T + g.start,)]
    by_lhs = {}
    for lhs, rhs in g.productions:
        by_lhs.setdefault(lhs, []).append(tuple(rhs))
    while frontier:
        nxt = []
        for form in frontier:
            i = next((k for k, s in enumerate(form) if s >= T), None)
            if i is None:
                out.add(form)
                continue
            for rhs in by_lhs.get(form[i] - T, []):
                f2 = form[:i] + rhs + form[i + 1:]
                if sum(1 for s in f2 if s < T) > maxlen or len(f2) > 2 * maxlen + 4:
                    continue
                if f2 not in seen:
                    seen.add(f2)
                    nxt.append(f2)
        frontier = nxt
    return out


def bar_hillel(g, n_nodes, gap, edges, start, accept):
    """R[X][u][v] = X derives some path u -> v, by fixpoint over boolean
    matrices (independent of the oracle's Earley parser)."""
    T, V = g.T, g.V
    N = n_nodes
    eps = np.eye(N, dtype=bool)
    for (u, v, lab) in edges:
        if lab < 0:
            eps[u, v] = True
    for _ in range(N):  # reflexive-transitive closure of epsilon edges
        e2 = (eps.astype(np.int32) @ eps.astype(np.int32)) > 0
        if (e2 == eps).all():
            break
        eps = e2
    term = np.zeros((T, N, N), dtype=bool)
    for (u, v, lab) in edges:
        if lab >= 0:
            term[lab, u, v] = True
    for u in range(N):
        if gap[u]:
            term[:, u, u] = True

    def mm(a, b):
        return (a.astype(np.int32) @ b.astype(np.int32)) > 0
    R_t = np.array([mm(mm(eps, term[a]), eps) for a in range(T)])
    R = np.zeros((V, N, N), dtype=bool)
    for _ in range(200):
        changed = False
        for lhs, rhs in g.productions:
            acc = eps.copy()
            for s in rhs:
                acc = mm(acc, R_t[s] if s < T else R[s - T])
                if not acc.any():
                    break
            new = R[lhs] | acc
            if (new != R[lhs]).any():
                R[lhs] = new
                changed = True
        if not changed:
            break
    return bool(R[g.start][start, accept])


def vocab_for(g, extra=()):
    chars = sorted(set(g.charset))
    toks = [c.encode() for c in chars] + [e.encode() for e in extra]
    return list(dict.fromkeys(toks))


def lexer_regex_module(g, text, flush=True):
    """Greedy lexer built from Python's `regex` partial matching: an
    independent implementation of the lexer reading."""
    regex = pytest.importorskip('regex')

    def py(rx):
        # same syntax as Python's except that ^ $ { } are plain bytes outside
        # classes; '.' excludes newline in both
        out, i, in_cls = [], 0, False
        while i < len(rx):
            c = rx[i]
            if c == '\\':
                out.append(rx[i:i + 2])
                i += 2
                continue
            if in_cls:
                if c == ']':
                    in_cls = False
                out.append(c)
            elif c == '[':
                in_cls = True
                out.append(c)
                if rx[i + 1:i + 2] == '^':
                    out.append('^')
                    i += 1
            elif c in '^${}':
                out.append('\\' + c)
            else:
                out.append(c)
            i += 1
        return ''.join(out)
    pats = [regex.compile(py(t.regex)) for t in g.terminals]
    run = []
    cur = ''
    i = 0
    while i < len(text):
        c = text[i]
        cand = cur + c
        if any(p.fullmatch(cand, partial=True) for p in pats):
            cur = cand
            i += 1
            continue
        acc = [k for k, p in enumerate(pats) if p.fullmatch(cur)] if cur else []
        if not acc:
            return None
        if not g.terminals[acc[0]].skip:
            run.append(acc[0])
        if not any(p.fullmatch(c, partial=True) for p in pats):
            return None
        cur = c  # restart from the initial state on c
        i += 1
    ends = flush
    if not flush and cur:  # before a gap: emit only a lexeme no byte can extend
        ends = not any(p.fullmatch(cur + chr(b), partial=True) for b in range(256) for p in pats)
    if ends and cur:
        acc = [k for k, p in enumerate(pats) if p.fullmatch(cur)]
        if not acc:
            return None
        if not g.terminals[acc[0]].skip:
            run.append(acc[0])
    return run


# ------------------------------------------------------------------ lexer
def test_lexer_golden_cases():
    g = expr()
    O = oracle.Oracle(g)
    names = {t.name: i for i, t in enumerate(g.terminals)}
    with open(os.path.join(HERE, 'golden', 'lexer_cases.txt')) as f:
        n = 0
        for line in f:
            if line.startswith('#') or not line.strip():
                continue
            text, flush, exp = line.rstrip('\n').split('\t')
            r = O.lex(text.encode(), 0, flush == '1')
            if exp == 'DEAD':
                assert r is None, text
            else:
                assert r is not None, text
                assert r[0] == [names[s] for s in exp.split()], text
            n += 1
    assert n >= 10


@pytest.mark.parametrize('gfun', [expr, words_grammar, G.json_grammar, G.smiles_grammar])
def test_lexer_matches_regex_module(gfun):
    g = gfun()
    O = oracle.Oracle(g)
    rng = np.random.default_rng(7)
    chars = sorted(set(g.charset))
    samples = [render(g, sample_derivation(g, rng, 8), rng) for _ in range(20)]
    texts = samples + [''.join(rng.choice(chars, size=int(rng.integers(1, 9)))) for _ in range(300)]
    for text in texts:
        for flush in (True, False):
            mine = O.lex(text.encode('latin-1'), 0, flush)
            ref = lexer_regex_module(g, text, flush)
            assert (mine is None) == (ref is None), (text, mine, ref)
            if mine is not None:
                assert mine[0] == ref, (text, mine, ref)


def test_lexer_one_byte_lookahead_dead_end():
    g = words_grammar()
    O = oracle.Oracle(g)
    names = {t.name: i for i, t in enumerate(g.terminals)}
    assert O.lex(b'<<=', 0, True)[0] == [names['SHLEQ']]
    assert O.lex(b'<', 0, True)[0] == [names['LT']]
    assert O.lex(b'<<', 0, True) is None          # "<<" is no lexeme; no backtracking
    assert O.lex(b'1.', 0, True) is None          # "1." cannot complete a NUM
    assert O.lex(b'ifx if', 0, True)[0] == [names['ID'], names['IF']]


# ------------------------------------------------------------------ Earley on strings
@pytest.mark.parametrize('gfun,maxlen', [(expr, 5), (tiny_paren, 7), (tiny_eps, 6), (tiny_nonrec, 3)])
def test_earley_equals_language_enumeration(gfun, maxlen):
    g = gfun()
    O = oracle.Oracle(g)
    L = language(g, maxlen)
    alphabet = [i for i, t in enumerate(g.terminals) if not t.skip]
    for m in range(0, maxlen + 1):
        for s in itertools.product(alphabet, repeat=m):
            assert O.accepts_terms(list(s)) == (s in L), s


# ------------------------------------------------------------------ graph validity
def random_partial(rng, vocab_n, n, p_mask):
    x = rng.integers(0, vocab_n, n).astype(np.int32)
    x[rng.random(n) < p_mask] = -1
    return x


@pytest.mark.parametrize('gfun,extra', [(expr, ['1+', '(2', '3)', '*(', ' 4']),
                                        (tiny_paren, ['((', 'a)', ' (']),
                                        (tiny_eps, ['xx', 'zy', 'yz']),
                                        (words_grammar, ['if', '<<', 'a ', '1.'])])
def test_earley_on_graph_equals_bar_hillel(gfun, extra):
    g = gfun()
    vocab = vocab_for(g, extra)
    O = oracle.Oracle(g, vocab)
    rng = np.random.default_rng(11)
    agree = 0
    for trial in range(120):
        n = int(rng.integers(0, 7))
        x = random_partial(rng, len(vocab), n, 0.35)
        nn, gap, edges, st, ac, dead = O.graph(x)
        if nn > 48:
            continue
        expect = False if dead else bar_hillel(g, nn, gap, edges, st, ac)
        assert O.valid(x) == expect, (x, edges)
        agree += 1
    assert agree >= 100


@pytest.mark.parametrize('gfun', [expr, tiny_paren, words_grammar, G.json_grammar])
def test_fully_masked_is_valid(gfun):
    g = gfun()
    O = oracle.Oracle(g, vocab_for(g))
    for n in (1, 2, 5):
        assert O.valid(np.full(n, -1, np.int32))


def test_unmasked_equals_membership_of_its_lexing():
    g = expr()
    vocab = vocab_for(g, ['1+', '(2', '3)', '*(', ' 4', '^-'])
    O = oracle.Oracle(g, vocab)
    L = language(g, 6)
    rng = np.random.default_rng(5)
    for _ in range(400):
        x = rng.integers(0, len(vocab), int(rng.integers(1, 5))).astype(np.int32)
        text = b''.join(vocab[t] for t in x).decode()
        run = lexer_regex_module(g, text, True)
        if run is None:
            assert not O.valid(x)
        elif len(run) <= 6:
            assert O.valid(x) == (tuple(run) in L), text


def test_prefix_then_gap_equals_viable_prefix():
    g = tiny_paren()
    vocab = vocab_for(g)
    O = oracle.Oracle(g, vocab)
    L = language(g, 9)
    prefixes = {s[:i] for s in L for i in range(len(s) + 1)}
    idx = {t.name: i for i, t in enumerate(g.terminals)}
    tokid = {v.decode(): i for i, v in enumerate(vocab)}
    for m in range(0, 5):
        for s in itertools.product('()a', repeat=m):
            x = np.array([tokid[c] for c in s] + [-1], np.int32)
            run = tuple(idx[c] for c in s)
            # with the trailing gap, the pending lexeme (none here: one-char
            # terminals) is absorbed; a viable prefix is a prefix of L(G)
            # restricted to sentences up to the enumerated length
            if run in prefixes:
                assert O.valid(x), s
            elif m <= 4:
                # any completion would be a sentence with this prefix; with
                # length <= 9 enumerated and this grammar, non-prefixes are
                # exactly the strings with more ')' than '(' somewhere or 'a'
                # directly before '(' / 'a' in an invalid position
                bal = 0
                ok = True
                for c in s:
                    bal += {'(': 1, ')': -1, 'a': 0}[c]
                    ok &= bal >= 0
                if not ok:
                    assert not O.valid(x), s


def test_one_sided_brute_force_over_fillings():
    g = expr()
    vocab = vocab_for(g, ['1+', '(2', '3)', '*('])
    O = oracle.Oracle(g, vocab)
    L = language(g, 7)
    rng = np.random.default_rng(3)
    hits = 0
    for _ in range(150):
        n = int(rng.integers(2, 5))
        x = random_partial(rng, len(vocab), n, 0.4)
        masks = np.flatnonzero(x < 0)
        if len(masks) == 0 or len(masks) > 2:
            continue
        v = O.valid(x)
        for fill in itertools.product(range(len(vocab)), repeat=len(masks)):
            y = x.copy()
            y[masks] = fill
            text = b''.join(vocab[t] for t in y).decode()
            run = lexer_regex_module(g, text, True)
            if run is not None and tuple(run) in L:
                assert v, (x, y)  # a concrete completion exists
                hits += 1
                break
    assert hits > 10


@pytest.mark.parametrize('name', ['expr-tiny', 'json-schema', 'smiles-256'])
def test_monotonicity_and_witness(name):
    w = make_workload(name, 42, batch=2, k=2, K=6)
    O = oracle.Oracle(w.grammar, w.vocab)
    for b in range(w.B):
        assert O.valid(w.x[b])                       # generated partial outputs are completable
        y = w.x[b].copy()
        for p in w.pos[b]:
            if w.witness[b, p] >= 0:
                y[p] = w.witness[b, p]
                assert O.valid(y)                    # the true tokens keep it completable
    v = O.validate_batch(w.x, w.pos, w.cand)
    # Valid(x (+) {(i, t), (j, u)}) implies Valid(x (+) {(i, t)})
    for b in range(w.B):
        for c1 in range(w.K):
            for c2 in range(w.K):
                y = w.x[b].copy()
                y[w.pos[b, 0]] = w.cand[b, 0, c1]
                y[w.pos[b, 1]] = w.cand[b, 1, c2]
                if O.valid(y):
                    assert v[b, 0, c1] == 1 and v[b, 1, c2] == 1


# ------------------------------------------------------------------ cover
COVER_GRAMMARS = {'expr': expr, 'tiny_paren': tiny_paren, 'tiny_eps': tiny_eps, 'json': G.json_grammar,
                  'smiles': G.smiles_grammar, 'clike-512': lambda: G.grammar_for('clike-512'),
                  'random-stress-1024': lambda: G.grammar_for('random-stress-1024')}


@pytest.mark.parametrize('gname', list(COVER_GRAMMARS))
def test_language_is_inside_the_cover(gname):
    """L(G) inside L(F_G) (the cover over-approximates, App. D) on 10,000
    sampled sentences per grammar."""
    g = COVER_GRAMMARS[gname]()
    O = oracle.Oracle(g)
    rng = np.random.default_rng(1)
    for _ in range(10000):
        terms = sample_derivation(g, rng, int(rng.integers(1, 25)))
        assert O.accepts_terms(terms)
        assert O.cover_accepts_terms(terms)


def test_cover_is_exact_without_recursion_or_sharing():
    g = tiny_nonrec()
    O = oracle.Oracle(g)
    alphabet = list(range(g.T))
    for m in range(0, 5):
        for s in itertools.product(alphabet, repeat=m):
            assert O.cover_accepts_terms(list(s)) == O.accepts_terms(list(s)), s


def test_cover_overapproximates_recursion():
    g = tiny_paren()
    O = oracle.Oracle(g)
    idx = {t.name: i for i, t in enumerate(g.terminals)}
    # exit(S) returns to every occurrence of S, so the ')' of S -> ( S ) S can
    # follow an S that no '(' opened
    s = [idx['a'], idx[')'], idx['a']]
    assert not O.accepts_terms(s)
    assert O.cover_accepts_terms(s)


@pytest.mark.parametrize('name', ['expr-tiny', 'json-schema'])
def test_exact_valid_implies_cover_valid(name):
    w = make_workload(name, 43, batch=2, k=2, K=8)
    O = oracle.Oracle(w.grammar, w.vocab)
    for b in range(w.B):
        for j in range(w.k):
            for c in range(w.K):
                y = w.x[b].copy()
                y[w.pos[b, j]] = w.cand[b, j, c]
                if O.valid(y):
                    assert O.cover_valid(y)


# ------------------------------------------------------------------ selection
def alg4_python(O, x, C):
    """Literal transcription of Alg. 4 with the oracle's tests as primitives."""
    def apply(x, S):
        y = x.copy()
        for (p, t) in S:
            y[p] = t
        return y

    def halves(S):
        h = (len(S) + 1) // 2
        return S[:h], S[h:]

    def relaxed(x, S):
        if len(S) <= 1:
            return []
        if O.cover_valid(apply(x, S)):
            return S
        L, R = halves(S)
        BL = relaxed(x, L)
        BR = relaxed(apply(x, BL), R)
        return BL + BR

    def shrink(x, S):
        if len(S) <= 1:
            return []
        if O.valid(apply(x, S)):
            return S
        L, R = halves(S)
        BLp = shrink(x, L)
        BRp = relaxed(apply(x, BLp), R)
        BRpp = shrink(apply(x, BLp), BRp)
        return BLp + BRpp
    return shrink(x, relaxed(x, C))


@pytest.mark.parametrize('name,seed', [('expr-tiny', 42), ('expr-tiny', 43), ('json-schema', 44),
                                       ('smiles-256', 42)])
def test_selection_matches_alg4_transcription(name, seed):
    w = make_workload(name, seed, batch=3 if name != 'expr-tiny' else 1, k=6 if name != 'expr-tiny' else None)
    O = oracle.Oracle(w.grammar, w.vocab)
    valid = O.validate_batch(w.x, w.pos, w.cand)
    tok, conf = oracle.pick_candidates(valid, w.cand, w.conf)
    sel = O.select(w.x, w.pos, tok, conf)
    for b in range(w.B):
        C = [(int(w.pos[b, j]), int(tok[b, j]), float(conf[b, j]), j) for j in range(w.k) if tok[b, j] >= 0]
        C.sort(key=lambda c: (-c[2], c[0]))
        Bsel = alg4_python(O, w.x[b], [(p, t) for (p, t, _, _) in C])
        slots = {j for (p, t, _, j) in C if (p, t) in set(Bsel)}
        assert set(np.flatnonzero(sel[b])) == slots
        assert len(slots) == 0 or len(slots) >= 2
        if slots:
            y = w.x[b].copy()
            for j in slots:
                y[w.pos[b, j]] = tok[b, j]
            assert O.valid(y)


def test_commit_writes_selected_tokens():
    x = np.full((2, 5), -1, np.int32)
    pos = np.array([[0, 3], [1, 2]], np.int32)
    tok = np.array([[7, 8], [9, 10]], np.int32)
    sel = np.array([[1, 0], [1, 1]], np.uint8)
    y = oracle.Oracle.commit(x, pos, tok, sel)
    assert y[0, 0] == 7 and y[0, 3] == -1 and y[1, 1] == 9 and y[1, 2] == 10


# ------------------------------------------------------------------ candidate set C
def load_select_cases():
    """tests/golden/select_cases.txt as (grammar, n, positions, tokens,
    confidences, expected selected, (cover tests, exact tests)) rows."""
    rows = []
    with open(os.path.join(HERE, 'golden', 'select_cases.txt')) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith('#'):
                continue
            gname, n, p, t, c, e, k = (s.strip() for s in line.split('|'))
            rows.append((gname, int(n), [int(a) for a in p.split()], [int(a) for a in t.split()],
                         [float(a) for a in c.split()], [int(a) for a in e.split()], tuple(int(a) for a in k.split())))
    return rows


def test_select_golden():
    """Alg. 4 (RelaxedSelect, then ExactShrink) on hand-derived cases: sizes
    one and two, a first half kept while the second fails, ties in confidence
    ordered by position, and a cover that over-accepts so that ExactShrink
    must shrink the relaxed set (and, in one case, down to nothing)."""
    grammars = {'nonrec': (tiny_nonrec(), [b'a', b'b', b'c', b'd', b'e']),
                'paren': (tiny_paren(), [b'(', b')', b'a', b'b'])}
    rows = load_select_cases()
    assert len(rows) >= 10
    for gname, n, pos, tok, conf, expect, tests in rows:
        spec, vocab = grammars[gname]
        O = oracle.Oracle(spec, vocab)
        x = np.full((1, n), -1, np.int32)
        sel = O.select(x, np.array([pos], np.int32), np.array([tok], np.int32), np.array([conf], np.float32))
        assert sel[0].tolist() == expect, (gname, pos, tok, conf, sel[0].tolist())
        assert O.last_select_counts == tests, (gname, pos, tok, conf, O.last_select_counts)


def test_fallback_golden():
    """Alg. 1's rejection fallback on hand-derived cases (tests/golden/
    fallback_cases.txt): commits in confidence order, rejections, positions
    committed by the selected batch skipped, ties by position then candidate
    index, n_t no larger than |B|; with the number of exact tests."""
    O = oracle.Oracle(tiny_nonrec(), [b'a', b'b', b'c', b'd', b'e'])
    cases = 0
    with open(os.path.join(HERE, 'golden', 'fallback_cases.txt')) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith('#'):
                continue
            xs, ps, ss, cs, fs, nt, ex, ef, et = (v.strip() for v in line.split('|'))
            x = np.array([[int(v) for v in xs.split()]], np.int32)
            pos = np.array([[int(v) for v in ps.split()]], np.int32)
            k = pos.shape[1]
            sel = np.array([[int(v) for v in ss.split()]], np.uint8)
            cand = np.array([int(v) for v in cs.split()], np.int32).reshape(1, k, -1)
            conf = np.array([float(v) for v in fs.split()], np.float32).reshape(1, k, -1)
            got_x, filled, nchk = O.fallback(x, pos, cand, conf, np.array([int(nt)], np.int32), sel)
            assert got_x[0].tolist() == [int(v) for v in ex.split()], line
            assert filled[0].tolist() == [int(v) for v in ef.split()], line
            assert nchk == int(et), (line, nchk)
            cases += 1
    assert cases >= 6


def load_pick_cases():
    """tests/golden/pick_cases.txt as (valid [R][4], conf [R][4], cand [R][4],
    expected token [R], expected confidence [R]); token of line r, index c is
    100 r + c."""
    rows = []
    with open(os.path.join(HERE, 'golden', 'pick_cases.txt')) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith('#'):
                continue
            v, c, t, e = (s.strip() for s in line.split('|'))
            rows.append(([int(a) for a in v.split()], [float(a) for a in c.split()], int(t), float(e)))
    R = len(rows)
    valid = np.array([r[0] for r in rows], np.uint8)
    conf = np.array([r[1] for r in rows], np.float32)
    cand = (100 * np.arange(R)[:, None] + np.arange(4)[None, :]).astype(np.int32)
    return valid, conf, cand, np.array([r[2] for r in rows], np.int32), np.array([r[3] for r in rows], np.float32)


@pytest.mark.parametrize('shape', [(1, 16), (4, 4), (2, 8)])
def test_pick_candidates_golden(shape):
    """Alg. 1's candidate set C on hand-derived cases: highest confidence among
    valid-bit-1 candidates, ties to the lowest index, overflow (2) never
    picked, none -> (-1, 0.0), -0.0 ties with 0.0 (the sign of the picked
    value is kept).  The rows are laid out as several batch shapes so that a
    transposed (sequence, position) index fails."""
    valid, conf, cand, etok, econf = load_pick_cases()
    B, k = shape
    assert B * k == len(etok)
    tok, cf = oracle.pick_candidates(valid.reshape(B, k, 4), cand.reshape(B, k, 4), conf.reshape(B, k, 4))
    np.testing.assert_array_equal(tok.reshape(-1), etok)
    np.testing.assert_array_equal(cf.reshape(-1).view(np.uint32), econf.view(np.uint32))


# ------------------------------------------------------------------ cover on partial outputs
def all_partials(vocab_n, n):
    for x in itertools.product(range(-1, vocab_n), repeat=n):
        yield np.array(x, np.int32)


def test_cover_valid_equals_valid_when_the_cover_is_exact():
    """tiny_nonrec's cover is exact (no recursion, no nonterminal used twice:
    L(F_G) = L(G), App. D.3), so on every partial output -- gaps included --
    the cover test 1[L(F_G) cap C_x != empty] and the exact test
    1[L(G) cap C_x != empty] of Sec. 3 must agree: both over- and
    under-acceptance of the cover's gap closure fail here."""
    g = tiny_nonrec()
    vocab = [b'a', b'b', b'c', b'd', b'e', b'ad', b'ab', b'ce']
    O = oracle.Oracle(g, vocab)
    n_valid = n_cover = 0
    for n in range(0, 5):
        for x in all_partials(len(vocab), n):
            v = O.valid(x)
            assert O.cover_valid(x) == v, x
            n_valid += v
            n_cover += 1
    rng = np.random.default_rng(9)
    for _ in range(3000):
        x = random_partial(rng, len(vocab), int(rng.integers(5, 9)), 0.4)
        assert O.cover_valid(x) == O.valid(x), x
    assert 0 < n_valid < n_cover


def _paren_runs(vocab, x):
    """Terminal view of a tiny_paren partial output whose tokens are made of
    the one-character terminals and skipped spaces: the fixed runs between
    gaps (as terminal-name strings) and whether each boundary is a gap."""
    segs, cur, gaps = [], '', []
    for t in x:
        if t < 0:
            if not gaps or not gaps[-1][1] or cur:
                segs.append(cur)
                gaps.append((len(segs) - 1, True))
                cur = ''
        else:
            cur += vocab[t].decode().replace(' ', '')
    segs.append(cur)
    return segs, sum(1 for _ in gaps)


def test_cover_valid_brute_force_over_gap_fillings():
    """tiny_paren (recursive; its cover over-accepts): the cover test of a
    partial output holds iff some filling of its gaps with terminal strings is
    accepted by the cover as a plain string.  The fillings are enumerated up
    to length 4 (one gap) or 3 (two gaps), over the terminals that occur in
    productions; the cover has few enough states that any state reachable
    across a gap is reachable within that length."""
    g = tiny_paren()
    vocab = [b'(', b')', b'a', b'b', b' ', b'((', b'a)', b' (']
    O = oracle.Oracle(g, vocab)
    idx = {t.name: i for i, t in enumerate(g.terminals)}
    fills = {L: [''.join(s) for m in range(L + 1) for s in itertools.product('()a', repeat=m)] for L in (3, 4)}
    cache = {}

    def cover_str(s):
        if s not in cache:
            cache[s] = O.cover_accepts_terms([idx[c] for c in s])
        return cache[s]

    checked = agree_true = 0
    for n in range(1, 5):
        for x in all_partials(len(vocab), n):
            segs, ngaps = _paren_runs(vocab, x)
            if ngaps > 2:
                continue
            L = 4 if ngaps <= 1 else 3
            if ngaps == 0:
                expect = cover_str(segs[0])
            elif ngaps == 1:
                expect = any(cover_str(segs[0] + f + segs[1]) for f in fills[L])
            else:
                expect = any(cover_str(segs[0] + f1 + segs[1] + f2 + segs[2])
                             for f1 in fills[L] for f2 in fills[L])
            assert O.cover_valid(x) == expect, (x, segs)
            checked += 1
            agree_true += expect
    assert checked > 3000 and 0 < agree_true < checked


# ------------------------------------------------------------------ Alg. 1's fallback
def fallback_python(O, x, pos, cand, conf, fill):
    """Alg. 1's sequential rejection loop transcribed with the oracle's exact
    test as the primitive: `fill` times, take the highest-confidence
    candidate at a still-masked position that was not rejected (ties:
    position, then candidate index); reject while x (+) c is invalid."""
    x = x.copy()
    order = sorted(((-float(conf[j, c]), int(pos[j]), c, j) for j in range(len(pos)) for c in range(cand.shape[1])))
    rejected = set()
    filled = {}
    for _ in range(fill):
        for (_, p, c, j) in order:
            if (j, c) in rejected or x[p] >= 0:
                continue
            y = x.copy()
            y[p] = cand[j, c]
            if O.valid(y):
                x[p] = cand[j, c]
                filled[j] = int(cand[j, c])
                break
            rejected.add((j, c))
        else:
            break
    return x, filled


@pytest.mark.parametrize('name,seed,kw', [('expr-tiny', 42, {}), ('expr-tiny', 44, dict(k=6, K=4)),
                                          ('json-schema', 42, dict(batch=2, k=6, K=6)),
                                          ('smiles-256', 43, dict(batch=2, k=6, K=5))])
def test_fallback_matches_alg1_transcription(name, seed, kw):
    w = make_workload(name, seed, **kw)
    O = oracle.Oracle(w.grammar, w.vocab)
    valid = O.validate_batch(w.x, w.pos, w.cand)
    tok, conf = oracle.pick_candidates(valid, w.cand, w.conf)
    sel = O.select(w.x, w.pos, tok, conf)
    x1 = O.commit(w.x, w.pos, tok, sel)
    n_target = np.full(w.B, w.k, np.int32)  # fill every proposed position if possible
    got_x, filled, nchk = O.fallback(x1, w.pos, w.cand, w.conf, n_target, sel)
    for b in range(w.B):
        ref_x, ref_f = fallback_python(O, x1[b], w.pos[b], w.cand[b], w.conf[b], int(n_target[b] - sel[b].sum()))
        np.testing.assert_array_equal(got_x[b], ref_x)
        assert {j: int(t) for j, t in enumerate(filled[b]) if t >= 0} == ref_f
    if (n_target - sel.sum(1)).sum() > 0:
        assert nchk > 0


@pytest.mark.parametrize('name,seed', [('expr-tiny', 43), ('json-schema', 45)])
def test_fallback_invariants(name, seed):
    """Every fallback commit fills a masked position and keeps the output
    completable (it was tested with all earlier commits applied); if fewer
    than asked were committed, every candidate left at a masked position is
    invalid for the final output (a rejected candidate stays invalid after
    later commits, by monotonicity of completability, App. D)."""
    w = make_workload(name, seed, batch=2, k=6, K=6)
    O = oracle.Oracle(w.grammar, w.vocab)
    n_target = np.array([3, 6], np.int32)
    got_x, filled, _ = O.fallback(w.x, w.pos, w.cand, w.conf, n_target)
    for b in range(w.B):
        committed = [j for j in range(w.k) if filled[b, j] >= 0]
        assert len(committed) <= n_target[b]
        for j in committed:
            assert w.x[b, w.pos[b, j]] < 0 and got_x[b, w.pos[b, j]] == filled[b, j]
        assert O.valid(got_x[b]) or not O.valid(w.x[b])
        if len(committed) < n_target[b]:
            for j in range(w.k):
                if got_x[b, w.pos[b, j]] >= 0:
                    continue
                for c in range(w.K):
                    y = got_x[b].copy()
                    y[w.pos[b, j]] = w.cand[b, j, c]
                    assert not O.valid(y)


# ------------------------------------------------------------------ witness checking
def test_graph_accepts_unmasked_rows_exactly_their_lexing():
    """A row without masks has one lexeme sequence (reading 1): the graph's
    path labels are exactly it (the independent regex-module lexer gives it);
    dropping, adding or changing one terminal is rejected."""
    g = expr()
    vocab = vocab_for(g, ['1+', '(2', '3)', '*(', ' 4', '^-'])
    O = oracle.Oracle(g, vocab)
    rng = np.random.default_rng(17)
    tested = 0
    for _ in range(300):
        x = rng.integers(0, len(vocab), int(rng.integers(1, 6))).astype(np.int32)
        text = b''.join(vocab[t] for t in x).decode()
        run = lexer_regex_module(g, text, True)
        if run is None:
            continue
        assert O.graph_accepts_terms(x, run), (text, run)
        if run:
            assert not O.graph_accepts_terms(x, run[:-1])
            changed = list(run)
            changed[0] = (changed[0] + 1) % g.T
            assert not O.graph_accepts_terms(x, changed)
        assert not O.graph_accepts_terms(x, list(run) + [0])
        tested += 1
    assert tested > 150


def test_graph_accepts_matches_gap_regex():
    """tiny_paren (one-character terminals, spaces skipped): the path labels
    of a partial output are its fixed runs with any terminal string in each
    gap -- a regular expression written from the gap model (Sec. 3), checked
    on every terminal string up to length 5."""
    import re
    g = tiny_paren()
    vocab = [b'(', b')', b'a', b'b', b' ', b'((', b'a)', b' (']
    O = oracle.Oracle(g, vocab)
    names = {t.name: i for i, t in enumerate(g.terminals)}
    sym = {names[c]: c for c in '()ab'}
    words = [''.join(s) for m in range(6) for s in itertools.product('()ab', repeat=m)]
    rng = np.random.default_rng(2)
    for _ in range(60):
        x = random_partial(rng, len(vocab), int(rng.integers(1, 5)), 0.4)
        segs, ngaps = _paren_runs(vocab, x)
        pattern = '.*'.join(re.escape(sg) for sg in segs)
        for wd in words:
            terms = [names[c] for c in wd]
            assert O.graph_accepts_terms(x, terms) == bool(re.fullmatch(pattern, wd)), (x, wd)

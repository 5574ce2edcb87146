"""GPU parity: the CUDA path (through the C-ABI) against the CPU oracle,
element by element on the same seeded inputs.  Validity bits and selected
sets are integer results, so the bar is bit-exact equality."""
import os

import numpy as np
import pytest

import oracle
from synth import make_workload

pytestmark = pytest.mark.gpu
NTHREADS = os.cpu_count() or 1


def _dev(a, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


def gpu_step(w, dev):
    import torch
    import paper_2606_00722_gb300 as epic
    g = epic.Grammar(w.grammar)
    t = epic.LexTable(g, w.vocab)
    x = _dev(w.x, dev)
    pos = _dev(w.pos, dev)
    cand = _dev(w.cand, dev)
    conf3 = _dev(w.conf, dev)
    valid = torch.empty(w.cand.shape, dtype=torch.uint8, device=dev)
    epic.validate_batch(g, t, x, pos, cand, valid)
    tok = torch.empty(w.pos.shape, dtype=torch.int32, device=dev)
    conf = torch.empty(w.pos.shape, dtype=torch.float32, device=dev)
    epic.pick_candidates(cand, conf3, valid, tok, conf)
    sel = torch.empty(w.pos.shape, dtype=torch.uint8, device=dev)
    epic.select_compatible_subset(g, t, x, pos, tok, conf, sel)
    epic.commit(x, pos, tok, sel)
    torch.cuda.synchronize()
    return dict(valid=valid.cpu().numpy(), tok=tok.cpu().numpy(), conf=conf.cpu().numpy(),
                sel=sel.cpu().numpy(), x=x.cpu().numpy(), stats=t.stats(), table=t, grammar=g)


CASES = [
    ('expr-tiny', 42, {}), ('expr-tiny', 43, {}), ('expr-tiny', 44, {}),
    ('json-schema', 42, dict(batch=4)), ('json-schema', 43, dict(batch=3, k=3)),
    ('smiles-256', 42, dict(batch=6, k=4)), ('smiles-256', 44, dict(batch=2, k=16, K=4)),
    ('clike-512', 42, dict(batch=1, k=2, K=4)),
]


@pytest.mark.parametrize('name,seed,kw', CASES)
def test_step_parity(cuda, name, seed, kw):
    w = make_workload(name, seed, **kw)
    O = oracle.Oracle(w.grammar, w.vocab)
    got = gpu_step(w, cuda)
    ref_valid = O.validate_batch(w.x, w.pos, w.cand, nthreads=NTHREADS)
    assert (got['valid'] != 2).all(), 'capacity overflow'
    np.testing.assert_array_equal(got['valid'], ref_valid)
    rtok, rconf = oracle.pick_candidates(ref_valid, w.cand, w.conf)
    np.testing.assert_array_equal(got['tok'], rtok)
    np.testing.assert_array_equal(got['conf'], rconf)
    ref_sel = O.select(w.x, w.pos, rtok, rconf)
    np.testing.assert_array_equal(got['sel'], ref_sel)
    np.testing.assert_array_equal(got['x'], O.commit(w.x, w.pos, rtok, ref_sel))
    assert got['stats']['checks'] == w.cand.size


@pytest.mark.parametrize('name,seed,kw', [('json-schema', 43, dict(batch=3, k=3)),
                                          ('clike-512', 42, dict(batch=2, k=4, K=4, n=160))])
def test_step_parity_descending_sweep(cuda, monkeypatch, name, seed, kw):
    """The CTA walks (forward charts of wide grammars, selection's exact
    tests) with the descending block sweep of the column closure instead of
    the warp-parallel one: the same least fixpoint, so the same bits."""
    monkeypatch.setenv('EPIC_GS_PARALLEL', '0')
    test_step_parity(cuda, name, seed, kw)


@pytest.mark.parametrize('name', ['expr-tiny', 'json-schema', 'smiles-256'])
def test_lex_table_runs_match_oracle(cuda, name):
    """Every token's run from the initial state, and the set of distinct runs
    over all lexer states, equal the oracle's lexing of the token's bytes."""
    w = make_workload(name, 42, batch=1, vocab_size=2000 if name != 'expr-tiny' else None)
    import paper_2606_00722_gb300 as epic
    g = epic.Grammar(w.grammar)
    t = epic.LexTable(g, w.vocab)
    end, ln, terms = t.entries()
    O = oracle.Oracle(w.grammar, w.vocab)
    nstates = O.n_lexer_states
    rng = np.random.default_rng(0)
    for tok in rng.choice(len(w.vocab), size=min(300, len(w.vocab)), replace=False):
        text = w.vocab[tok]
        r0 = O.lex(text, 0, run_only=True)
        assert (r0 is None) == (end[tok, 0] == 0xFFFF)
        if r0 is not None:
            assert list(terms[tok, 0, :ln[tok, 0]]) == r0[0]
        mine = {tuple(terms[tok, q, :ln[tok, q]]) for q in range(end.shape[1]) if end[tok, q] != 0xFFFF}
        ref = set()
        for q in range(nstates):
            r = O.lex(text, q, run_only=True)
            if r is not None:
                ref.add(tuple(r[0]))
        assert mine == ref, (text, mine ^ ref)


@pytest.mark.parametrize('shape', [(1, 16), (4, 4), (2, 8)])
def test_pick_golden(cuda, shape):
    """k_pick (Alg. 1's candidate set C) on the hand-derived golden cases,
    bit for bit including the sign of a picked -0.0."""
    import torch
    import paper_2606_00722_gb300 as epic
    from test_oracle_pins import load_pick_cases
    valid, conf, cand, etok, econf = load_pick_cases()
    B, k = shape
    tok = torch.empty((B, k), dtype=torch.int32, device=cuda)
    cf = torch.empty((B, k), dtype=torch.float32, device=cuda)
    epic.pick_candidates(_dev(cand.reshape(B, k, 4), cuda), _dev(conf.reshape(B, k, 4), cuda),
                         _dev(valid.reshape(B, k, 4), cuda), tok, cf)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(tok.cpu().numpy().reshape(-1), etok)
    np.testing.assert_array_equal(cf.cpu().numpy().reshape(-1).view(np.uint32), econf.view(np.uint32))


@pytest.mark.parametrize('name,seed,kw,fill', [
    ('expr-tiny', 42, {}, 8), ('expr-tiny', 45, dict(k=6, K=4), 6),
    ('json-schema', 43, dict(batch=3, k=6, K=6), 6), ('smiles-256', 44, dict(batch=3, k=6, K=5), 4),
    ('clike-512', 42, dict(batch=1, k=2, K=4, n=128), 2),
])
def test_decode_step_with_fallback(cuda, name, seed, kw, fill):
    """One whole step (validate, pick, select, commit, then Alg. 1's rejection
    fallback for the commits still wanted) against the oracle's, bit-exact:
    validity bits, selected batch, fallback commits and the final x."""
    import torch
    import paper_2606_00722_gb300 as epic
    w = make_workload(name, seed, **kw)
    O = oracle.Oracle(w.grammar, w.vocab)
    n_target = np.full(w.B, fill, np.int32)
    g = epic.Grammar(w.grammar)
    t = epic.LexTable(g, w.vocab)
    x = _dev(w.x, cuda)
    bufs = dict(valid=torch.empty(w.cand.shape, dtype=torch.uint8, device=cuda),
                tok=torch.empty(w.pos.shape, dtype=torch.int32, device=cuda),
                conf=torch.empty(w.pos.shape, dtype=torch.float32, device=cuda),
                selected=torch.empty(w.pos.shape, dtype=torch.uint8, device=cuda),
                filled=torch.empty(w.pos.shape, dtype=torch.int32, device=cuda))
    epic.decode_step(g, t, x, _dev(w.pos, cuda), _dev(w.cand, cuda), _dev(w.conf, cuda), _dev(n_target, cuda), bufs)
    torch.cuda.synchronize()
    st = t.stats()
    ref_valid = O.validate_batch(w.x, w.pos, w.cand, nthreads=NTHREADS)
    rtok, rconf = oracle.pick_candidates(ref_valid, w.cand, w.conf)
    ref_sel = O.select(w.x, w.pos, rtok, rconf)
    x1 = O.commit(w.x, w.pos, rtok, ref_sel)
    ref_x, ref_filled, nchk = O.fallback(x1, w.pos, w.cand, w.conf, n_target, ref_sel)
    np.testing.assert_array_equal(bufs['valid'].cpu().numpy(), ref_valid)
    np.testing.assert_array_equal(bufs['selected'].cpu().numpy(), ref_sel)
    np.testing.assert_array_equal(bufs['filled'].cpu().numpy(), ref_filled)
    np.testing.assert_array_equal(x.cpu().numpy(), ref_x)
    # (decode_step hands the fallback the step's validity bits: candidates
    # whose bit is 0 are rejected untested, with the same result)
    assert st['fallback_commits'] == int((ref_filled >= 0).sum())
    # without the bits every candidate is tested, as in the oracle's loop
    # (a round also tests the candidates after its commit)
    x2 = _dev(x1, cuda)
    filled2 = torch.empty(w.pos.shape, dtype=torch.int32, device=cuda)
    t.stats(reset=True)
    epic.fallback_commit(g, t, x2, _dev(w.pos, cuda), _dev(w.cand, cuda), _dev(w.conf, cuda), _dev(n_target, cuda),
                         _dev(ref_sel, cuda), filled2)
    torch.cuda.synchronize()
    st2 = t.stats()
    np.testing.assert_array_equal(filled2.cpu().numpy(), ref_filled)
    np.testing.assert_array_equal(x2.cpu().numpy(), ref_x)
    # the rounds test at least the candidates the sequential loop tests
    assert st2['fallback_checks'] >= nchk


def _step_with_table(w, dev, lazy_capacity):
    import torch
    import paper_2606_00722_gb300 as epic
    g = epic.Grammar(w.grammar)
    t = epic.LexTable(g, w.vocab, lazy_capacity=lazy_capacity)
    x = _dev(w.x, dev)
    pos = _dev(w.pos, dev)
    cand = _dev(w.cand, dev)
    conf3 = _dev(w.conf, dev)
    bufs = dict(valid=torch.empty(w.cand.shape, dtype=torch.uint8, device=dev),
                tok=torch.empty(w.pos.shape, dtype=torch.int32, device=dev),
                conf=torch.empty(w.pos.shape, dtype=torch.float32, device=dev),
                selected=torch.empty(w.pos.shape, dtype=torch.uint8, device=dev),
                filled=torch.empty(w.pos.shape, dtype=torch.int32, device=dev))
    epic.decode_step(g, t, x, pos, cand, conf3, _dev(np.full(w.B, w.k, np.int32), dev), bufs)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in bufs.items()}, x.cpu().numpy(), t.stats()


@pytest.mark.parametrize('name,seed,kw', [
    ('expr-tiny', 42, {}), ('json-schema', 42, dict(batch=4)), ('smiles-256', 43, dict(batch=6, k=4)),
    ('clike-512', 42, dict(batch=1, k=2, K=4, n=128)),
])
def test_lazy_lex_memo_equals_dense_table(cuda, name, seed, kw):
    """Alg. 2's lexing memo filled on first use (no dense table): whole steps
    identical to those with the dense table, with a memo large enough to hold
    every entry used and with one too small for most (entries then computed
    without being stored); the counters give the memo's hit rate."""
    w = make_workload(name, seed, **kw)
    ref, ref_x, ref_st = _step_with_table(w, cuda, None)
    assert ref_st['lex_lookups'] > 0 and ref_st['lex_misses'] == 0
    for cap in (1 << 20, 64):
        got, got_x, st = _step_with_table(w, cuda, cap)
        for key in ('valid', 'selected', 'filled'):
            np.testing.assert_array_equal(got[key], ref[key])
        np.testing.assert_array_equal(got_x, ref_x)
        assert st['lex_lookups'] == ref_st['lex_lookups']
        assert 0 < st['lex_misses'] <= st['lex_lookups']
        if cap == 64:
            assert st['lex_uncached'] > 0
        else:
            # a lookup that finds its entry still being computed by another
            # thread may compute it itself (bounded wait): rare, not a miss of capacity
            assert st['lex_uncached'] <= st['lex_lookups'] // 100 and st['lex_misses'] < st['lex_lookups']

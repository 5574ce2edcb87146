"""GPU edge cases against the oracle: boundary positions, single-mask runs
between spans (the candidate joins both neighbours' lexemes), fully masked
rows, one-token rows, dead lexings, K = 1 / k = 1, bad inputs, empty batches,
and sampled checks of the full benchmark batch."""
import os

import numpy as np
import pytest

import oracle
from synth import grammars as G
from synth import make_workload

pytestmark = pytest.mark.gpu
NTHREADS = os.cpu_count() or 1


def words_grammar():
    b = G._Builder('words')
    b.lit('if', 'IF')
    b.lit('<<=', 'SHLEQ')
    b.lit('<', 'LT')
    b.term('ID', '[a-z]+', ('word', 'ab', 'ab', 1, 3))
    b.term('NUM', '[0-9]+(\\.[0-9]+)?', ('digits', 1, 2))
    b.term('WS', '[ ]+', ('ws',), skip=True)
    b.rule('S', 'S X', 'IF ID LT NUM')
    b.rule('X', 'IF', 'SHLEQ', 'LT', 'ID', 'NUM')
    return b.build('S', 'abfi<=0123. ')


def run_gpu(spec, vocab, x, pos, cand, dev):
    import torch
    import paper_2606_00722_gb300 as epic
    g = epic.Grammar(spec)
    t = epic.LexTable(g, vocab)
    xt = torch.from_numpy(np.ascontiguousarray(x, np.int32)).to(dev)
    pt = torch.from_numpy(np.ascontiguousarray(pos, np.int32)).to(dev)
    ct = torch.from_numpy(np.ascontiguousarray(cand, np.int32)).to(dev)
    valid = torch.full(cand.shape, 9, dtype=torch.uint8, device=dev)
    epic.validate_batch(g, t, xt, pt, ct, valid)
    torch.cuda.synchronize()
    return valid.cpu().numpy(), t.stats()


def rows_with_all_positions(rng, vocab_n, n, p_mask, reps):
    """Rows and, for each row, every masked position proposed once (k = all)."""
    xs, ps = [], []
    while len(xs) < reps:
        x = rng.integers(0, vocab_n, n).astype(np.int32)
        x[rng.random(n) < p_mask] = -1
        m = np.flatnonzero(x < 0)
        if len(m) == 0:
            continue
        xs.append(x)
        ps.append(m)
    k = max(len(p) for p in ps)
    X = np.stack(xs)
    P = np.zeros((reps, k), np.int32)
    for i, p in enumerate(ps):
        P[i, :len(p)] = p
        P[i, len(p):] = p[0]  # repeat a masked position (results compared per slot)
    return X, P


@pytest.mark.parametrize('gname', ['expr', 'words'])
def test_every_position_shape(cuda, gname):
    """All masked positions of short random rows: runs of length one between
    spans, positions 0 and n-1, leading and trailing gaps, dead lexings."""
    spec = G.expr_grammar() if gname == 'expr' else words_grammar()
    extra = ['1+', '(2', '3)', '*(', ' 4', '^-'] if gname == 'expr' else ['if', '<<', 'a ', '1.', 'f<', '<<=']
    vocab = list(dict.fromkeys([c.encode() for c in sorted(set(spec.charset))] + [e.encode() for e in extra]))
    rng = np.random.default_rng(17)
    for n in (1, 2, 3, 5, 9):
        X, P = rows_with_all_positions(rng, len(vocab), n, 0.45, 6)
        cand = rng.integers(0, len(vocab), (X.shape[0], P.shape[1], 5)).astype(np.int32)
        got, _ = run_gpu(spec, vocab, X, P, cand, cuda)
        ref = oracle.Oracle(spec, vocab).validate_batch(X, P, cand, nthreads=NTHREADS)
        np.testing.assert_array_equal(got, ref)


def test_fully_masked_rows_and_K1(cuda):
    spec = G.json_grammar()
    w = make_workload('json-schema', 44, batch=2, k=3, K=1)
    x = np.full_like(w.x, -1)
    got, _ = run_gpu(spec, w.vocab, x, w.pos, w.cand, cuda)
    ref = oracle.Oracle(spec, w.vocab).validate_batch(x, w.pos, w.cand)
    np.testing.assert_array_equal(got, ref)


def test_bad_inputs_give_zero_and_are_counted(cuda):
    w = make_workload('expr-tiny', 42)
    x = w.x.copy()
    pos = w.pos.copy()
    cand = w.cand.copy()
    pos[0, 0] = int(np.flatnonzero(x[0] >= 0)[0])      # not a masked position
    cand[0, 1, 0] = len(w.vocab) + 5                    # token id out of range
    got, st = run_gpu(w.grammar, w.vocab, x, pos, cand, cuda)
    assert (got[0, 0] == 0).all()
    assert got[0, 1, 0] == 0
    assert st['bad_inputs'] >= w.K + 1
    # every other check is unaffected
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x, w.pos, w.cand)
    np.testing.assert_array_equal(got[0, 2:], ref[0, 2:])


def test_empty_batches_are_no_ops(cuda):
    import torch
    import paper_2606_00722_gb300 as epic
    w = make_workload('expr-tiny', 42)
    g = epic.Grammar(w.grammar)
    t = epic.LexTable(g, w.vocab)
    x = torch.from_numpy(w.x).to(cuda)
    pos = torch.zeros((1, 0), dtype=torch.int32, device=cuda)
    cand = torch.zeros((1, 0, 4), dtype=torch.int32, device=cuda)
    valid = torch.zeros((1, 0, 4), dtype=torch.uint8, device=cuda)
    epic.validate_batch(g, t, x, pos, cand, valid)
    torch.cuda.synchronize()
    assert t.stats()['checks'] == 0


def test_selection_edges(cuda):
    """k = 1 (a single candidate is never a batch), no valid candidate, and a
    NaN confidence (bad input: nothing selected)."""
    import torch
    import paper_2606_00722_gb300 as epic
    w = make_workload('json-schema', 42, batch=3, k=4)
    g = epic.Grammar(w.grammar)
    t = epic.LexTable(g, w.vocab)
    x = torch.from_numpy(w.x).to(cuda)
    pos = torch.from_numpy(w.pos).to(cuda)
    tok = np.full((3, 4), -1, np.int32)
    conf = np.zeros((3, 4), np.float32)
    tok[0, 0] = w.witness[0, w.pos[0, 0]]
    conf[0, 0] = 0.5                                    # row 0: a single candidate
    for j in range(4):                                  # row 2: NaN confidence
        tok[2, j] = w.witness[2, w.pos[2, j]]
        conf[2, j] = np.float32('nan') if j == 1 else 0.1 * (j + 1)
    sel = torch.full((3, 4), 9, dtype=torch.uint8, device=cuda)
    epic.select_compatible_subset(g, t, x, pos, torch.from_numpy(tok).to(cuda),
                                  torch.from_numpy(conf).to(cuda), sel)
    torch.cuda.synchronize()
    s = sel.cpu().numpy()
    assert (s == 0).all()
    ref = oracle.Oracle(w.grammar, w.vocab).select(w.x[:2], w.pos[:2], tok[:2], conf[:2])
    np.testing.assert_array_equal(s[:2], ref)


def test_full_benchmark_batch_parity(cuda):
    """The benchmark's own batch (json-schema, 16 x 256 tokens, k = 4, K = 16),
    in the launch configuration bench.py times: every check against the
    oracle."""
    w = make_workload('json-schema', 42)
    got, st = run_gpu(w.grammar, w.vocab, w.x, w.pos, w.cand, cuda)
    assert st['overflow'] == 0
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x, w.pos, w.cand, nthreads=NTHREADS)
    np.testing.assert_array_equal(got, ref)


def test_smiles_full_size_sampled(cuda):
    """smiles-256 at its full size (256 x 256 tokens, k = 16, K = 16): all
    65,536 checks on the GPU, a seeded sample of rows checked by the oracle."""
    w = make_workload('smiles-256', 42)
    got, st = run_gpu(w.grammar, w.vocab, w.x, w.pos, w.cand, cuda)
    assert st['overflow'] == 0
    rows = np.random.default_rng(0).choice(w.B, size=6, replace=False)
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x[rows], w.pos[rows], w.cand[rows],
                                                          nthreads=NTHREADS)
    np.testing.assert_array_equal(got[rows], ref)
    # property at any size: a valid single update implies a completable x
    O = oracle.Oracle(w.grammar, w.vocab)
    for b in rows[:2]:
        assert O.valid(w.x[b]) or not got[b].any()

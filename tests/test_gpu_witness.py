"""Witness extraction for failure recovery (Sec. 4.4) on the GPU.  Several
completions can be right, so each witness is checked for what makes it one:
its lexeme sequence is in L(G) (the oracle's Earley recognizer) and is a path
of the partial output's graph (the oracle's graph, gaps reading anything);
rows that are not completable get none."""
import os

import numpy as np
import pytest

import oracle
from synth import make_workload

from test_gpu_edges import rows_with_all_positions, words_grammar

pytestmark = pytest.mark.gpu


def _witness(spec, vocab, x, dev, cap=None):
    import torch
    import paper_2606_00722_gb300 as epic
    g = epic.Grammar(spec)
    t = epic.LexTable(g, vocab)
    n = x.shape[1]
    cap = cap or 16 * n + 64
    xt = torch.from_numpy(np.ascontiguousarray(x, np.int32)).to(dev)
    terms = torch.full((x.shape[0], cap), -7, dtype=torch.int32, device=dev)
    lens = torch.full((x.shape[0],), -9, dtype=torch.int32, device=dev)
    epic.extract_witness(g, t, xt, terms, lens)
    torch.cuda.synchronize()
    return terms.cpu().numpy(), lens.cpu().numpy(), t.stats()


def _check_rows(spec, vocab, x, terms, lens, O):
    import paper_2606_00722_gb300 as epic
    n_wit = 0
    for b in range(x.shape[0]):
        valid = O.valid(x[b])
        if not valid:
            assert lens[b] == -1, (b, lens[b])
            continue
        assert lens[b] >= 0, (b, lens[b])
        w = terms[b, :lens[b]] & (epic.GAP_BIT - 1)
        assert O.accepts_terms(list(w)), (b, w)
        assert O.graph_accepts_terms(x[b], list(w)), (b, w)
        n_wit += 1
    return n_wit


@pytest.mark.parametrize('name,seed,kw', [
    ('expr-tiny', 42, dict(batch=6)), ('json-schema', 42, dict(batch=6)), ('smiles-256', 43, dict(batch=8)),
    ('clike-512', 42, dict(batch=3, n=160)),
])
def test_witness_of_generated_rows(cuda, name, seed, kw):
    """Completable rows of the workloads (and the same rows with their first
    fixed token replaced by a random one, mostly not completable)."""
    w = make_workload(name, seed, **kw)
    rng = np.random.default_rng(3)
    x = w.x.copy()
    broken = w.x.copy()
    for b in range(w.B):
        fixed = np.flatnonzero(broken[b] >= 0)
        if len(fixed):
            broken[b, fixed[0]] = rng.integers(0, len(w.vocab))
    rows = np.concatenate([x, broken])
    terms, lens, st = _witness(w.grammar, w.vocab, rows, cuda)
    O = oracle.Oracle(w.grammar, w.vocab)
    assert _check_rows(w.grammar, w.vocab, rows, terms, lens, O) >= w.B
    assert st['witness_failures'] == 0


def test_witness_of_short_random_rows(cuda):
    """Short random partial outputs of a grammar with multi-character
    lexemes and a one-byte-lookahead dead end: every completable one gets a
    witness, the others none."""
    spec = words_grammar()
    vocab = list(dict.fromkeys([c.encode() for c in sorted(set(spec.charset))] +
                               [e.encode() for e in ['if', '<<', 'a ', '1.', 'f<', '<<=']]))
    rng = np.random.default_rng(8)
    X, _ = rows_with_all_positions(rng, len(vocab), 9, 0.45, 24)
    terms, lens, st = _witness(spec, vocab, X, cuda)
    O = oracle.Oracle(spec, vocab)
    _check_rows(spec, vocab, X, terms, lens, O)
    assert (lens >= 0).any() and (lens == -1).any()
    assert st['witness_failures'] == 0


def test_witness_capacity_is_reported(cuda):
    """A capacity too small for the witness reports -2, never a cut sequence."""
    w = make_workload('json-schema', 43, batch=2)
    terms, lens, _ = _witness(w.grammar, w.vocab, w.x, cuda, cap=3)
    assert (lens == -2).all()

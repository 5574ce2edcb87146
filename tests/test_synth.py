"""The seeded synthetic workloads (CPU): shapes, grammar sizes, mask fractions
and candidate distributions of the five benchmark configurations, determinism
by seed, and the internal consistency the parity tests rely on."""
import numpy as np
import pytest

from synth import make_workload

# name: (B, n, k, K, vocab, mask fraction, terminals, nonterminals, productions)
CONFIGS = {
    'expr-tiny': (1, 32, 8, 8, 256, 0.25, 10, 6, 14),
    'json-schema': (16, 256, 4, 16, 32768, 0.40, 40, 30, 65),
    'clike-512': (32, 512, 8, 32, 65536, 0.50, 100, 150, 500),
    'random-stress-1024': (64, 1024, 16, 32, 126000, 0.60, 128, 400, 1500),
    'smiles-256': (256, 256, 16, 16, 126000, 0.50, 43, 35, 104),
}


@pytest.mark.parametrize('name', sorted(CONFIGS))
def test_workload_matches_its_configuration(name):
    B, n, k, K, V, mask, T, NT, P = CONFIGS[name]
    w = make_workload(name, 42)
    assert (w.B, w.n, w.k, w.K, len(w.vocab)) == (B, n, k, K, V)
    assert w.x.shape == (B, n) and w.pos.shape == (B, k) and w.cand.shape == (B, k, K) == w.conf.shape
    assert abs(float((w.x < 0).mean()) - mask) < 0.02
    g = w.grammar
    assert g.T == T and len({lhs for lhs, _ in g.productions}) == NT and len(g.productions) == P
    # proposed positions: distinct masked positions of the row
    for b in range(B):
        assert (w.x[b, w.pos[b]] < 0).all()
        assert len(set(w.pos[b].tolist())) == k
    assert ((w.cand >= 0) & (w.cand < V)).all()
    assert all(len(set(w.cand[b, j].tolist())) == K for b in range(B) for j in range(k))  # distinct candidates
    # candidate confidences: probabilities of one distribution per position
    assert np.isfinite(w.conf).all() and (w.conf > 0).all() and (w.conf.sum(axis=2) <= 1.0 + 1e-5).all()
    # the row's completion agrees with every fixed token
    fixed = w.x >= 0
    assert (w.witness[fixed] == w.x[fixed]).all()
    assert all(0 < len(t) for t in w.vocab)


def test_workloads_are_determined_by_the_seed():
    a, b, c = make_workload('json-schema', 42), make_workload('json-schema', 42), make_workload('json-schema', 43)
    for key in ('x', 'pos', 'cand', 'conf'):
        np.testing.assert_array_equal(getattr(a, key), getattr(b, key))
    assert not np.array_equal(a.x, c.x)
    assert a.vocab == b.vocab


def test_a_smaller_batch_keeps_the_first_rows():
    """Profiling runs use a prefix of the benchmark batch: the same rows and
    proposed positions (so the same forward charts)."""
    full, small = make_workload('clike-512', 42), make_workload('clike-512', 42, batch=2)
    np.testing.assert_array_equal(full.x[:2], small.x)
    np.testing.assert_array_equal(full.pos[:2], small.pos)

"""epic_validate_batch_noalloc -- validation without any device allocation,
for callers that cannot call cudaMalloc (a serving process whose device
memory is all reserved by its own pool, or a decode loop that must not take
cudaMalloc's synchronization).  Its results must equal epic_validate_batch's
(bit-exact: validity bits are integers), call after call, although every
call reuses the library's one fixed scratch array.

This file is collected last so that a run stopping at the first failure has
already run every other test."""
import numpy as np
import pytest

from synth import make_workload

pytestmark = pytest.mark.gpu


def _run(fn, w, dev):
    import torch
    import paper_2606_00722_gb300 as epic
    g = epic.Grammar(w.grammar)
    t = epic.LexTable(g, w.vocab)
    x = torch.from_numpy(w.x).to(dev)
    pos = torch.from_numpy(w.pos).to(dev)
    cand = torch.from_numpy(w.cand).to(dev)
    valid = torch.full(w.cand.shape, 7, dtype=torch.uint8, device=dev)
    fn(g, t, x, pos, cand, valid)
    torch.cuda.synchronize()
    return valid.cpu().numpy()


def test_noalloc_equals_validate_batch_on_two_calls_in_a_row(cuda):
    import paper_2606_00722_gb300 as epic
    # two different batches back to back: the second call must not see the
    # first one's leftovers in the shared scratch array
    for name, seed, kw in [('json-schema', 42, dict(batch=4)), ('smiles-256', 43, dict(batch=4, k=4))]:
        w = make_workload(name, seed, **kw)
        ref = _run(epic.validate_batch, w, cuda)
        got = _run(epic.validate_batch_noalloc, w, cuda)
        assert (ref != 2).all() and (got != 2).all()
        np.testing.assert_array_equal(got, ref)


def test_noalloc_wide_items_short_rows_global_stage(cuda):
    """A grammar whose item sets exceed 32 words (clike-512: 150
    nonterminals, 500 productions) keeps its rows in the global part of the
    fixed array, which the call clears itself; two different short batches
    back to back must both equal epic_validate_batch (which answers these
    checks by region)."""
    import paper_2606_00722_gb300 as epic
    for seed, kw in [(42, dict(batch=1, k=2, K=4, n=48)), (43, dict(batch=2, k=2, K=3, n=64))]:
        w = make_workload('clike-512', seed, **kw)
        ref = _run(epic.validate_batch, w, cuda)
        got = _run(epic.validate_batch_noalloc, w, cuda)
        assert (ref != 2).all() and (got != 2).all()
        np.testing.assert_array_equal(got, ref)


def test_noalloc_rejects_long_rows_of_wide_grammars(cuda):
    """Wide item sets on rows longer than 128 tokens are refused with
    EPIC_ERR_CAPACITY before anything is enqueued (the output is untouched)."""
    import torch
    import paper_2606_00722_gb300 as epic
    w = make_workload('clike-512', 42, batch=1, k=1, K=2, n=200)
    g = epic.Grammar(w.grammar)
    t = epic.LexTable(g, w.vocab)
    x = torch.from_numpy(w.x).to(cuda)
    pos = torch.from_numpy(w.pos).to(cuda)
    cand = torch.from_numpy(w.cand).to(cuda)
    valid = torch.full(w.cand.shape, 7, dtype=torch.uint8, device=cuda)
    with pytest.raises(epic.EpicError) as e:
        epic.validate_batch_noalloc(g, t, x, pos, cand, valid)
    assert e.value.status == 6  # EPIC_ERR_CAPACITY
    torch.cuda.synchronize()
    assert (valid.cpu().numpy() == 7).all()


def test_noalloc_on_a_side_stream_then_stats(cuda):
    """A call on a stream other than the table's previous one: the
    statistics read afterwards must include its checks (epic_get_stats waits
    for the stream the last call used)."""
    import torch
    import paper_2606_00722_gb300 as epic
    w = make_workload('json-schema', 44, batch=3, k=2, K=4)
    g = epic.Grammar(w.grammar)
    t = epic.LexTable(g, w.vocab)
    x = torch.from_numpy(w.x).to(cuda)
    pos = torch.from_numpy(w.pos).to(cuda)
    cand = torch.from_numpy(w.cand).to(cuda)
    valid = torch.full(w.cand.shape, 7, dtype=torch.uint8, device=cuda)
    torch.cuda.synchronize()
    t.stats(reset=True)
    side = torch.cuda.Stream()
    with torch.cuda.stream(side):
        epic.validate_batch_noalloc(g, t, x, pos, cand, valid, stream=side)
    st = t.stats()
    assert st['checks'] == w.cand.size
    torch.cuda.synchronize()
    assert set(np.unique(valid.cpu().numpy())) <= {0, 1}


def test_noalloc_rejects_argument_errors(cuda):
    import ctypes
    import paper_2606_00722_gb300 as epic
    lib = epic.load()
    assert lib.epic_validate_batch_noalloc(None, None, None, 1, 1, None, 1, None, 1, None, None) == 1

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


def test_noalloc_rejects_argument_errors(cuda):
    import ctypes
    import paper_2606_00722_gb300 as epic
    lib = epic.load()
    assert lib.epic_validate_batch_noalloc(None, None, None, 1, 1, None, 1, None, 1, None, None) == 1

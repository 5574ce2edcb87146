"""Failure paths on the GPU, in the safe form: every device loop is bounded,
and a check or a sequence that runs out of a capacity gives up inside its
bounds and reports (value 2 in d_valid, stats.overflow), never faulting or
hanging.  The capacities are made tiny through the library's workspace knobs
so that the limits are reached on ordinary inputs."""
import os

import numpy as np
import pytest

import oracle
from synth import make_workload

from test_gpu_edges import run_gpu

pytestmark = pytest.mark.gpu
NTHREADS = os.cpu_count() or 1


def test_whole_walk_overflow_reports_two(cuda, monkeypatch):
    """Whole-graph walks with room for 40 chart entries: checks whose chart
    needs more report 2 and are counted; every other bit equals the oracle."""
    monkeypatch.setenv('EPIC_REGION', '0')
    monkeypatch.setenv('EPIC_ENTRIES_PER_WALK', '40')
    w = make_workload('json-schema', 42, batch=2, k=3, K=6, n=64)
    got, st = run_gpu(w.grammar, w.vocab, w.x, w.pos, w.cand, cuda)
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x, w.pos, w.cand, nthreads=NTHREADS)
    ovf = got == 2
    assert ovf.any(), 'the tiny workspace should overflow some checks'
    assert st['overflow'] == int(ovf.sum())
    np.testing.assert_array_equal(got[~ovf], ref[~ovf])
    assert set(np.unique(got)) <= {0, 1, 2}


def test_region_chart_overflow_falls_back_to_whole_walks(cuda, monkeypatch):
    """Per-sequence forward charts with room for 300 entries: sequences whose
    chart does not fit walk their checks whole instead, with the same bits
    as the oracle (nothing is reported as overflow: the whole walks have
    their own room)."""
    monkeypatch.setenv('EPIC_REGION', '1')
    monkeypatch.setenv('EPIC_SEQ_ENTRIES', '300')
    w = make_workload('json-schema', 43, batch=3, k=3, K=5, n=96)
    got, st = run_gpu(w.grammar, w.vocab, w.x, w.pos, w.cand, cuda)
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x, w.pos, w.cand, nthreads=NTHREADS)
    assert st['overflow'] == 0
    np.testing.assert_array_equal(got, ref)


@pytest.mark.parametrize('forward_cta', ['0', '1'])
def test_both_limits_at_once(cuda, monkeypatch, forward_cta):
    """Forward charts and whole walks both too small (either forward kernel):
    the checks report 2, none is silently answered."""
    monkeypatch.setenv('EPIC_REGION', '1')
    monkeypatch.setenv('EPIC_FORWARD_CTA', forward_cta)
    monkeypatch.setenv('EPIC_SEQ_ENTRIES', '200')
    monkeypatch.setenv('EPIC_ENTRIES_PER_WALK', '30')
    w = make_workload('json-schema', 44, batch=2, k=2, K=4, n=80)
    got, st = run_gpu(w.grammar, w.vocab, w.x, w.pos, w.cand, cuda)
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x, w.pos, w.cand, nthreads=NTHREADS)
    ovf = got == 2
    assert st['overflow'] == int(ovf.sum())
    np.testing.assert_array_equal(got[~ovf], ref[~ovf])
    assert ovf.any()

"""The C-ABI library builds for sm_103a, loads, and exports every entry point
that include/*.h declares; without a GPU the calls fail loudly (no CPU
fallback)."""
import glob
import os
import re

import pytest

import paper_2606_00722_gb300 as epic

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, 'include', '*.h')):
        src = open(h).read()
        src = re.sub(r'/\*.*?\*/', '', src, flags=re.S)
        for m in re.finditer(r'^[A-Za-z_][\w \*]*?\b(epic_\w+)\s*\(', src, flags=re.M):
            names.add(m.group(1))
    return names


def test_library_exports_every_declared_symbol():
    path = epic.build()
    lib = epic.load(path)
    names = declared_functions()
    assert len(names) >= 12
    for n in sorted(names):
        assert hasattr(lib, n), n
    assert set(epic.EXPORTS) <= names


def test_status_strings():
    lib = epic.load(epic.build())
    for s in range(8):
        assert lib.epic_status_string(s)


def test_no_cpu_fallback_without_gpu():
    import torch
    if torch.cuda.is_available():
        pytest.skip('a GPU is present')
    from synth import grammar_for
    with pytest.raises(epic.EpicError) as e:
        epic.Grammar(grammar_for('expr-tiny'))
    assert e.value.status == 5  # EPIC_ERR_CUDA


def test_host_side_argument_errors():
    """Argument errors are detected on the host, before any device work."""
    import ctypes as C
    lib = epic.load(epic.build())
    out = C.c_void_p()
    assert lib.epic_grammar_create(None, C.byref(out)) == 1
    d = epic.epic._Desc()
    d.n_terminals = 0  # no terminals
    assert lib.epic_grammar_create(C.byref(d), C.byref(out)) == 1
    # null objects and negative sizes
    assert lib.epic_validate_batch(None, None, None, 1, 1, None, 1, None, 1, None, None) == 1
    assert lib.epic_select_compatible_subset(None, None, None, 1, 1, None, 1, None, None, None, None) == 1
    assert lib.epic_commit(None, -1, 1, None, 1, None, None, None) == 1
    assert lib.epic_pick_candidates(None, None, None, 1, 1, 1, None, None, None) == 1
    # empty batches are no-ops that touch nothing
    assert lib.epic_commit(None, 0, 5, None, 3, None, None, None) == 0
    assert lib.epic_pick_candidates(None, None, None, 0, 4, 4, None, None, None) == 0


def test_stats_struct_matches_header():
    """The binding's epic_stats mirror has the header's fields, in order, all
    uint64 (the library copies the whole struct)."""
    src = open(os.path.join(ROOT, 'include', 'epic.h')).read()
    body = re.search(r'typedef struct \{(.*?)\} epic_stats;', src, flags=re.S).group(1)
    body = re.sub(r'/\*.*?\*/', '', body, flags=re.S)
    fields = re.findall(r'uint64_t\s+(\w+)\s*;', body)
    from paper_2606_00722_gb300.epic import _Stats
    assert [f for f, _ in _Stats._fields_] == fields
    import ctypes
    assert ctypes.sizeof(_Stats) == 8 * len(fields)

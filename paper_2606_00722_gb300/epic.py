"""Thin ctypes binding of the EPIC C-ABI (``include/epic.h``).

Argument marshalling only: every step of the hot path runs in the CUDA
library ``_build/libepic.so``.  Device buffers are passed as torch CUDA
tensors (their data pointers), host buffers as numpy arrays.  If the library
is missing or no CUDA device is usable the calls raise -- there is no CPU
fallback.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
# translation units, compiled in parallel and linked into one library
_SRC = [os.path.join(_HERE, 'csrc', f) for f in
        ('epic.cu', 'kernels_walk.cu', 'kernels_select.cu', 'region_forward.cu', 'region_good.cu',
         'region_check_sm.cu', 'region_check_global.cu', 'peak.cu', 'witness.cu', 'grammar.cpp')]
_DEPS = _SRC + [os.path.join(_HERE, 'csrc', f) for f in
                ('grammar.h', 'device.cuh', 'walk.cuh', 'cover.cuh', 'skeleton.cuh', 'warpwalk.cuh', 'packs.cuh',
                 'seqpack.cuh', 'launch.h', 'region.cuh', 'region_check.cuh', 'gscols.cuh')] + \
    [os.path.join(_HERE, '..', 'include', 'epic.h'), os.path.join(_HERE, '..', 'include', 'epic_measure.h')]
LIB_PATH = os.path.join(_HERE, '_build', 'libepic.so')
ARCH_FLAGS = ['-gencode', 'arch=compute_103a,code=sm_103a']
COMPILE_FLAGS = ARCH_FLAGS + ['-lineinfo', '-O3', '-std=c++17', '-Xcompiler', '-fPIC']
NVCC_FLAGS = COMPILE_FLAGS + ['-shared']  # one-command form: nvcc NVCC_FLAGS sources -o lib

OK, ERR_INVALID_ARG, ERR_GRAMMAR, ERR_LEXER, ERR_OOM, ERR_CUDA, ERR_CAPACITY, ERR_TIMEOUT = range(8)


class EpicError(RuntimeError):
    def __init__(self, status, where):
        super().__init__('%s: %s (status %d)' % (where, _status_string(status), status))
        self.status = status


def build(force: bool = False, verbose: bool = False, extra_flags=()) -> str:
    """Compile the CUDA library for sm_103a (nvcc cross-compiles without a
    GPU): every translation unit in parallel, then one link."""
    os.makedirs(os.path.dirname(LIB_PATH), exist_ok=True)
    newest = max(os.path.getmtime(p) for p in _DEPS)
    if force or not os.path.exists(LIB_PATH) or os.path.getmtime(LIB_PATH) < newest:
        tag = '%d' % os.getpid()
        objs, procs = [], []
        for src in _SRC:
            obj = os.path.join(os.path.dirname(LIB_PATH), os.path.basename(src) + '.%s.o' % tag)
            cmd = ['nvcc'] + COMPILE_FLAGS + list(extra_flags) + ['-c', src, '-o', obj]
            if verbose:
                print(' '.join(cmd))
            procs.append((subprocess.Popen(cmd), cmd))
            objs.append(obj)
        failed = [cmd for p, cmd in procs if p.wait() != 0]
        try:
            if failed:
                raise subprocess.CalledProcessError(1, failed[0])
            tmp = LIB_PATH + '.tmp' + tag
            cmd = ['nvcc'] + ARCH_FLAGS + ['-shared'] + objs + ['-o', tmp]
            if verbose:
                print(' '.join(cmd))
            subprocess.check_call(cmd)
            os.replace(tmp, LIB_PATH)
        finally:
            for o in objs:
                if os.path.exists(o):
                    os.remove(o)
    return LIB_PATH


class _Stats(C.Structure):
    _fields_ = [(n, C.c_uint64) for n in ('checks', 'valid', 'overflow', 'bad_inputs', 'columns',
                                          'entries', 'cover_checks', 'exact_checks', 'selected',
                                          'region_checks', 'validate_kernels', 'fallback_checks',
                                          'fallback_commits', 'lex_lookups', 'lex_misses', 'lex_uncached',
                                          'witness_failures', 'fallback_rounds')]


class _Desc(C.Structure):
    _fields_ = [('n_terminals', C.c_int32), ('terminal_regex', C.POINTER(C.c_char_p)),
                ('terminal_skip', C.POINTER(C.c_uint8)), ('n_nonterminals', C.c_int32),
                ('start', C.c_int32), ('n_productions', C.c_int32), ('lhs', C.POINTER(C.c_int32)),
                ('rhs_off', C.POINTER(C.c_int32)), ('rhs', C.POINTER(C.c_int32))]


_lib = None
EXPORTS = ('epic_grammar_create', 'epic_grammar_destroy', 'epic_grammar_lexer_states',
           'epic_lexer_table_build', 'epic_lexer_table_build_lazy', 'epic_lexer_table_destroy',
           'epic_lexer_table_copy',
           'epic_validate_batch', 'epic_validate_batch_noalloc',
           'epic_pick_candidates', 'epic_select_compatible_subset', 'epic_commit', 'epic_fallback_commit',
           'epic_extract_witness',
           'epic_get_stats', 'epic_status_string', 'epic_measure_int_peak', 'epic_last_kernel_times')


def load(path: str | None = None):
    """Load the library (raises OSError if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    lib = C.CDLL(path or LIB_PATH)
    vp, i32, u8p, i32p = C.c_void_p, C.c_int32, C.POINTER(C.c_uint8), C.POINTER(C.c_int32)
    lib.epic_status_string.restype = C.c_char_p
    lib.epic_status_string.argtypes = [C.c_int]
    lib.epic_grammar_create.argtypes = [C.POINTER(_Desc), C.POINTER(vp)]
    lib.epic_grammar_destroy.argtypes = [vp]
    lib.epic_grammar_lexer_states.argtypes = [vp]
    lib.epic_grammar_lexer_states.restype = i32
    lib.epic_lexer_table_build.argtypes = [vp, i32p, u8p, i32, vp, C.POINTER(vp)]
    lib.epic_lexer_table_build_lazy.argtypes = [vp, i32p, u8p, i32, C.c_int64, vp, C.POINTER(vp)]
    lib.epic_lexer_table_destroy.argtypes = [vp]
    lib.epic_lexer_table_copy.argtypes = [vp, i32, i32, vp, C.c_size_t]
    lib.epic_validate_batch.argtypes = [vp, vp, vp, i32, i32, vp, i32, vp, i32, vp, vp]
    lib.epic_validate_batch_noalloc.argtypes = [vp, vp, vp, i32, i32, vp, i32, vp, i32, vp, vp]
    lib.epic_pick_candidates.argtypes = [vp, vp, vp, i32, i32, i32, vp, vp, vp]
    lib.epic_select_compatible_subset.argtypes = [vp, vp, vp, i32, i32, vp, i32, vp, vp, vp, vp]
    lib.epic_commit.argtypes = [vp, i32, i32, vp, i32, vp, vp, vp]
    lib.epic_fallback_commit.argtypes = [vp, vp, vp, i32, i32, vp, i32, vp, vp, i32, vp, vp, vp, vp, vp]
    lib.epic_extract_witness.argtypes = [vp, vp, vp, i32, i32, vp, i32, vp, vp]
    lib.epic_get_stats.argtypes = [vp, C.POINTER(_Stats), C.c_size_t, C.c_int]
    lib.epic_measure_int_peak.argtypes = [C.POINTER(C.c_double), C.POINTER(C.c_double), vp]
    lib.epic_measure_int_peak.restype = C.c_int
    lib.epic_last_kernel_times.argtypes = [vp, C.POINTER(C.c_float), C.POINTER(C.c_char_p), C.c_int]
    lib.epic_last_kernel_times.restype = C.c_int
    _lib = lib
    return lib


def _status_string(s):
    try:
        return load().epic_status_string(int(s)).decode()
    except OSError:
        return 'status %d' % s


def _check(status, where):
    if status != OK:
        raise EpicError(status, where)


def _ptr(t):
    """Device pointer of a torch tensor (or an int address)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_cuda:
        raise ValueError('expected a CUDA tensor')
    if not t.is_contiguous():
        raise ValueError('expected a contiguous tensor')
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


class Grammar:
    """epic_grammar_create / epic_grammar_destroy."""

    def __init__(self, spec):
        lib = load()
        T = spec.T
        self._regs = (C.c_char_p * T)(*[t.regex.encode('latin-1') for t in spec.terminals])
        self._skip = np.array([1 if t.skip else 0 for t in spec.terminals], np.uint8)
        lhs, off, rhs = spec.rhs_flat()
        self._arrs = (lhs, off, rhs if rhs.size else np.zeros(1, np.int32))
        d = _Desc(T, self._regs, self._skip.ctypes.data_as(C.POINTER(C.c_uint8)), spec.V, spec.start,
                  len(spec.productions), lhs.ctypes.data_as(C.POINTER(C.c_int32)),
                  off.ctypes.data_as(C.POINTER(C.c_int32)),
                  self._arrs[2].ctypes.data_as(C.POINTER(C.c_int32)))
        h = C.c_void_p()
        _check(lib.epic_grammar_create(C.byref(d), C.byref(h)), 'epic_grammar_create')
        self.h = h
        self.spec = spec

    @property
    def lexer_states(self):
        return load().epic_grammar_lexer_states(self.h)

    def close(self):
        if getattr(self, 'h', None):
            load().epic_grammar_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class LexTable:
    """epic_lexer_table_build / epic_lexer_table_destroy."""

    def __init__(self, grammar: Grammar, vocab, stream=None, lazy_capacity: int | None = None):
        """lazy_capacity: build lazily (epic_lexer_table_build_lazy) with a
        memo of that many entries, instead of the dense table."""
        lib = load()
        lens = np.array([len(t) for t in vocab], np.int64)
        off = np.zeros(len(vocab) + 1, np.int32)
        off[1:] = np.cumsum(lens)
        data = np.frombuffer(b''.join(vocab), np.uint8).copy()
        h = C.c_void_p()
        if lazy_capacity is None:
            _check(lib.epic_lexer_table_build(grammar.h, off.ctypes.data_as(C.POINTER(C.c_int32)),
                                              data.ctypes.data_as(C.POINTER(C.c_uint8)), len(vocab),
                                              _stream(stream), C.byref(h)), 'epic_lexer_table_build')
        else:
            _check(lib.epic_lexer_table_build_lazy(grammar.h, off.ctypes.data_as(C.POINTER(C.c_int32)),
                                                   data.ctypes.data_as(C.POINTER(C.c_uint8)), len(vocab),
                                                   int(lazy_capacity), _stream(stream), C.byref(h)),
                   'epic_lexer_table_build_lazy')
        self.h = h
        self.grammar = grammar
        self.vocab = len(vocab)

    def entries(self, first: int = 0, count: int | None = None):
        """Lex-table rows as (end [count][Q] uint16, len [count][Q] uint8,
        terms [count][Q][13] uint8); end 0xFFFF is DEAD."""
        count = self.vocab - first if count is None else count
        Q = self.grammar.lexer_states
        raw = np.zeros((count, Q, 16), np.uint8)
        _check(load().epic_lexer_table_copy(self.h, first, count, raw.ctypes.data, raw.nbytes),
               'epic_lexer_table_copy')
        end = raw[:, :, 0].astype(np.uint16) | (raw[:, :, 1].astype(np.uint16) << 8)
        return end, raw[:, :, 2], raw[:, :, 3:16]

    def stats(self, reset: bool = False) -> dict:
        s = _Stats()
        _check(load().epic_get_stats(self.h, C.byref(s), C.sizeof(s), int(reset)), 'epic_get_stats')
        return {n: int(getattr(s, n)) for n, _ in _Stats._fields_}

    def kernel_times(self) -> dict:
        """epic_last_kernel_times: {kernel name: ms} of the last
        validate_batch and select_compatible_subset calls on this table
        (synchronizes)."""
        ms = (C.c_float * 8)()
        names = (C.c_char_p * 8)()
        n = load().epic_last_kernel_times(self.h, ms, names, 8)
        if n < 0:
            raise EpicError(ERR_CUDA, 'epic_last_kernel_times')
        return {names[i].decode(): float(ms[i]) for i in range(n)}

    def close(self):
        if getattr(self, 'h', None):
            load().epic_lexer_table_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def measure_int_peak(stream=None):
    """epic_measure_int_peak: (word operations per second, kernel ms) of the
    integer pipe on the current device (the roofline denominator of the
    walks)."""
    rate, ms = C.c_double(0), C.c_double(0)
    r = load().epic_measure_int_peak(C.byref(rate), C.byref(ms), _stream(stream))
    if r != 0:
        raise EpicError(r, 'epic_measure_int_peak')
    return rate.value, ms.value


def validate_batch(g: Grammar, t: LexTable, x, pos, cand, valid, stream=None):
    B, n = x.shape
    k = pos.shape[1]
    K = cand.shape[2]
    _check(load().epic_validate_batch(g.h, t.h, _ptr(x), B, n, _ptr(pos), k, _ptr(cand), K, _ptr(valid),
                                      _stream(stream)), 'epic_validate_batch')


def validate_batch_noalloc(g: Grammar, t: LexTable, x, pos, cand, valid, stream=None):
    """epic_validate_batch_noalloc: the same checks with no device allocation
    (scratch in a fixed array inside the library), for callers whose device
    memory is all reserved by their own pool or whose decode loop must not
    call cudaMalloc.  Calls on one device must not overlap on the GPU."""
    B, n = x.shape
    k = pos.shape[1]
    K = cand.shape[2]
    _check(load().epic_validate_batch_noalloc(g.h, t.h, _ptr(x), B, n, _ptr(pos), k, _ptr(cand), K,
                                              _ptr(valid), _stream(stream)), 'epic_validate_batch_noalloc')


def pick_candidates(cand, cand_conf, valid, tok, conf, stream=None):
    B, k, K = cand.shape
    _check(load().epic_pick_candidates(_ptr(cand), _ptr(cand_conf), _ptr(valid), B, k, K, _ptr(tok),
                                       _ptr(conf), _stream(stream)), 'epic_pick_candidates')


def select_compatible_subset(g: Grammar, t: LexTable, x, pos, tok, conf, selected, stream=None):
    B, n = x.shape
    k = pos.shape[1]
    _check(load().epic_select_compatible_subset(g.h, t.h, _ptr(x), B, n, _ptr(pos), k, _ptr(tok),
                                                _ptr(conf), _ptr(selected), _stream(stream)),
           'epic_select_compatible_subset')


def commit(x, pos, tok, selected, stream=None):
    B, n = x.shape
    k = pos.shape[1]
    _check(load().epic_commit(_ptr(x), B, n, _ptr(pos), k, _ptr(tok), _ptr(selected), _stream(stream)),
           'epic_commit')


def fallback_commit(g: Grammar, t: LexTable, x, pos, cand, cand_conf, n_target, selected, filled, stream=None,
                    valid=None):
    """epic_fallback_commit: Alg. 1's sequential rejection fallback (selected
    may be None for an empty batch B; valid, the single-candidate bits of x
    before the commits, lets it skip candidates that would fail)."""
    B, n = x.shape
    k = pos.shape[1]
    K = cand.shape[2]
    _check(load().epic_fallback_commit(g.h, t.h, _ptr(x), B, n, _ptr(pos), k, _ptr(cand), _ptr(cand_conf), K,
                                       _ptr(n_target), _ptr(selected), _ptr(valid), _ptr(filled),
                                       _stream(stream)), 'epic_fallback_commit')


def decode_step(g: Grammar, t: LexTable, x, pos, cand, cand_conf, n_target, bufs, stream=None):
    """One denoising step's constraint work (Alg. 1 after the model's
    proposal): validate every (position, candidate), pick C, select and commit
    the relaxed-compatible batch B (Alg. 4), then fill the commits still
    wanted by the rejection fallback.  bufs holds the device outputs: valid
    [B][k][K] uint8, tok [B][k] int32, conf [B][k] float32, selected [B][k]
    uint8, filled [B][k] int32.  Only sequences the C-ABI calls; asynchronous."""
    validate_batch(g, t, x, pos, cand, bufs['valid'], stream)
    pick_candidates(cand, cand_conf, bufs['valid'], bufs['tok'], bufs['conf'], stream)
    select_compatible_subset(g, t, x, pos, bufs['tok'], bufs['conf'], bufs['selected'], stream)
    commit(x, pos, bufs['tok'], bufs['selected'], stream)
    fallback_commit(g, t, x, pos, cand, cand_conf, n_target, bufs['selected'], bufs['filled'], stream,
                    valid=bufs['valid'])


GAP_BIT = 1 << 16  # a witness terminal produced inside a mask run


def extract_witness(g: Grammar, t: LexTable, x, terms, lengths, stream=None):
    """epic_extract_witness: terms [B][cap] int32 (terminal | GAP_BIT when a
    gap produces it), lengths [B] int32 (-1: not completable, -2: capacity)."""
    B, n = x.shape
    _check(load().epic_extract_witness(g.h, t.h, _ptr(x), B, n, _ptr(terms), terms.shape[1], _ptr(lengths),
                                       _stream(stream)), 'epic_extract_witness')

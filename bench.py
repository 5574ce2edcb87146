"""Benchmark of one denoising step's constraint work on GB300.

A step = epic_validate_batch + epic_pick_candidates +
epic_select_compatible_subset + epic_commit + epic_fallback_commit over one
batch of the workload: every proposed (position, candidate) pair checked, the
relaxed-compatible subset selected, checked jointly and committed, then Alg.
1's rejection fallback fills the commits still wanted (n_t = k per sequence).
Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   (the CPU oracle on the same config)

Multi-GPU (torchrun, one rank per GPU): replicas -- every rank runs its own
seeded batch of the same shape; there is no data-path collective.
"""
import argparse
import json
import os
import subprocess
import tempfile
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

# ncu summaries of the kernels' DRAM traffic (profiles/traffic_<kernel>_<workload>.txt): used only while the
# kernel's sources hash to the value recorded with the counters
KERNEL_SOURCES = {
    'k_validate_warp': ['kernels_walk.cu', 'warpwalk.cuh', 'device.cuh', 'packs.cuh'],
    'k_forward_gs': ['region_forward.cu', 'gscols.cuh', 'skeleton.cuh', 'walk.cuh', 'device.cuh', 'seqpack.cuh'],
    'k_forward': ['region_forward.cu', 'warpwalk.cuh', 'device.cuh', 'seqpack.cuh'],
    'k_good': ['region_good.cu', 'gscols.cuh', 'device.cuh', 'seqpack.cuh'],
    'k_check': ['region_check.cuh', 'region_check_sm.cu', 'region_check_global.cu', 'warpwalk.cuh', 'device.cuh'],
}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument('--gpus', type=int, default=1)
    ap.add_argument('--steps', type=int, default=5)
    ap.add_argument('--warmup', type=int, default=3)
    # clike-512 (32 x 512, k 8, K 32) is the largest workload whose steps fit
    # a bench run of minutes; random-stress-1024 (64 x 1024, k 16, K 32) runs
    # with --workload random-stress-1024 at several minutes per step
    ap.add_argument('--workload', default='clike-512')
    ap.add_argument('--impl', default='epic', choices=['epic', 'reference'])
    ap.add_argument('--seed', type=int, default=42)
    ap.add_argument('--cpu-seconds', type=float, default=15.0)
    ap.add_argument('--ref-seconds', type=float, default=20.0,
                    help='host time of one step of the reference arm (the oracle)')
    ap.add_argument('--no-cpu-baseline', action='store_true')
    ap.add_argument('--k', type=int, default=None, help='proposed positions per sequence (sweep)')
    ap.add_argument('--batch', type=int, default=None, help='sequences per batch (smaller cases for profiling)')
    ap.add_argument('--lazy-lex', type=int, default=None, metavar='CAP',
                    help='lexing memo filled on use (Alg. 2) with CAP entries instead of the dense table')
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get('RANK', '0'))
    world = int(os.environ.get('WORLD_SIZE', '1'))
    local = int(os.environ.get('LOCAL_RANK', '0'))
    return rank, world, local


def peaks():
    p = os.path.join(ROOT, 'MEASURED_PEAKS.json')
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, 'measured'
    return {'hbm_gbs': 6800.0, 'bf16_tflops': 1900.0, 'sm_max_mhz': 2070.0}, 'fallback'


class Clocks:
    """nvidia-smi sampling during the timed region."""

    def __init__(self, index):
        self.index = index
        self.proc = None
        # the raw samples go to EPIC_CLOCKS_CSV when set, else to a temporary file
        self.path = os.environ.get('EPIC_CLOCKS_CSV') or os.path.join(
            tempfile.gettempdir(), 'epic_bench_clocks_%d.csv' % os.getpid())

    def __enter__(self):
        os.makedirs(os.path.dirname(os.path.abspath(self.path)), exist_ok=True)
        q = ('index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,'
             'clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,'
             'clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap')
        try:
            self.f = open(self.path, 'w')
            self.proc = subprocess.Popen(['nvidia-smi', '-i', str(self.index), '--query-gpu=' + q,
                                          '--format=csv,noheader,nounits', '-lms', '200'],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if not self.proc or not os.path.exists(self.path):
            return {'sm_mhz': None, 'sm_max_mhz': None, 'reasons': ['unsampled']}
        sm, mx, reasons = [], [], set()
        names = ['hw_slowdown', 'hw_thermal_slowdown', 'sw_thermal_slowdown', 'sw_power_cap']
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(',')]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for nm, v in zip(names, parts[5:9]):
                    if v.lower() == 'active':
                        reasons.add(nm)
        if not sm:
            return {'sm_mhz': None, 'sm_max_mhz': None, 'reasons': ['unsampled']}
        return {'sm_mhz': float(np.median(sm)), 'sm_max_mhz': max(mx), 'reasons': sorted(reasons),
                'samples': len(sm)}


def kernel_sha(kernel):
    """Hash of a kernel's source files (tells whether recorded counters still
    describe the current build)."""
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES.get(kernel, []):
        with open(os.path.join(ROOT, 'paper_2606_00722_gb300', 'csrc', f), 'rb') as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel, workload):
    """DRAM bytes per launch from profiles/traffic_<kernel>_<workload>.txt
    (key: value lines), or None if absent or recorded for other sources."""
    path = os.path.join(ROOT, 'profiles', 'traffic_%s_%s.txt' % (kernel, workload))
    if not os.path.exists(path):
        return None
    rec = {}
    with open(path) as f:
        for line in f:
            if ':' in line and not line.startswith('#'):
                k, v = line.split(':', 1)
                rec[k.strip()] = v.strip()
    if rec.get('source_sha16') != kernel_sha(kernel):
        return None
    try:
        return float(rec['dram_bytes_per_launch'])
    except (KeyError, ValueError):
        return None


def census(workload, batch):
    """The oracle's chart census of the workload (tests/golden/census_*.json,
    written by tests/golden/make_census.py): item words per entry, and the
    (node, origin) pairs of the forward charts of x over the batch (sample
    mean times the batch) and, where counted, of every check's own chart."""
    path = os.path.join(ROOT, 'tests', 'golden', 'census_%s.json' % workload)
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f)
    per = d.get('per_seq', [])
    out = {'words': d['words'], 'file': os.path.relpath(path, ROOT)}
    if per:
        out['forward_pairs'] = float(np.mean([r['pairs'] for r in per])) * batch
        out['forward_sample'] = '%d of %d sequences' % (len(per), batch)
    if 'checks_pairs' in d:
        out['checks_pairs'] = float(d['checks_pairs'])
    return out


def cpu_baseline(w, seconds):
    """The oracle as it stands on the host cores, on a bounded sample of the
    workload's checks (whole sequences, all their candidates, in order)."""
    import oracle
    cores = os.cpu_count() or 1
    if w.n >= 1024:
        return cpu_baseline_bounded(w, seconds, cores)
    O = oracle.Oracle(w.grammar, w.vocab)
    # proposed positions in batch order, all K candidates of one per call (on
    # every core), until the budget is spent
    t0 = time.perf_counter()
    done = 0
    calls = 0
    while calls < w.B * w.k and (time.perf_counter() - t0) < seconds:
        b, j = divmod(calls, w.k)
        O.validate_batch(w.x[b:b + 1], w.pos[b:b + 1, j:j + 1], w.cand[b:b + 1, j:j + 1], nthreads=cores)
        done += w.K
        calls += 1
    dt = time.perf_counter() - t0
    # the same oracle on one core: the first sequence's positions in turn (all
    # their candidates per call), for at most a fifth of the budget
    t1 = time.perf_counter()
    one = 0
    for j in range(w.k):
        if one and time.perf_counter() - t1 > seconds / 5:
            break
        O.validate_batch(w.x[:1], w.pos[:1, j:j + 1], w.cand[:1, j:j + 1], nthreads=1)
        one += w.K
    dt1 = time.perf_counter() - t1
    return {'value': done / dt, 'unit': 'checks/s', 'cores': cores, 'kind': 'oracle',
            'sample': '%d of %d proposed positions in batch order (%d checks), oracle validate_batch on %d '
                      'threads, %.1f s' % (calls, w.B * w.k, done, cores, dt),
            'value_1core': one / dt1,
            'sample_1core': '%d checks of the first sequence, one position per call on 1 thread, %.1f s'
                            % (one, dt1)}


def _one_check(args):
    name, seed, k, b, j, c = args
    import oracle
    from synth import make_workload
    w = make_workload(name, seed, k=k)
    O = oracle.Oracle(w.grammar, w.vocab)
    O.validate_batch(w.x[b:b + 1], w.pos[b:b + 1, j:j + 1], w.cand[b:b + 1, j:j + 1, c:c + 1])
    return 1


def cpu_baseline_bounded(w, seconds, cores):
    """Rows of a thousand tokens: one oracle check takes longer than the whole
    budget (its chart runs to the end of the row), so one check per core runs
    for at most `seconds` in worker processes; the rate is the finished checks
    over the time, or, when none finishes, an upper bound of one check per
    core over the budget."""
    import multiprocessing as mp
    jobs = [(w.name, w.seed, w.k, 0, j % w.k, j // w.k) for j in range(cores)]
    ctx = mp.get_context('spawn')
    t0 = time.perf_counter()
    pool = ctx.Pool(cores)
    res = [pool.apply_async(_one_check, (a,)) for a in jobs]
    done = 0
    deadline = t0 + seconds
    for r in res:
        try:
            done += r.get(timeout=max(0.0, deadline - time.perf_counter()))
        except mp.TimeoutError:
            pass
    dt = time.perf_counter() - t0
    pool.terminate()
    pool.join()
    bound = done == 0
    value = (cores if bound else done) / dt
    return {'value': value, 'unit': 'checks/s', 'cores': cores, 'kind': 'oracle',
            'bound': 'upper' if bound else None,
            'sample': '%d checks of sequence 0 (one per core, %d positions) for at most %.0f s: %d finished%s'
                      % (cores, min(cores, w.k), seconds, done,
                         '; value is one check per core over the budget, an upper bound' if bound else '')}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from synth import make_workload
    w = make_workload(args.workload, args.seed, k=args.k, batch=args.batch)
    import oracle
    O = oracle.Oracle(w.grammar, w.vocab)
    cores = os.cpu_count() or 1
    # each step: a bounded sample of the workload -- the proposed positions
    # in batch order (continuing from the previous step), all K candidates of
    # one position per call on every core, until the step has run
    # --ref-seconds -- so that the whole run stays within minutes
    per_step, per_checks = [], []
    nxt = 0
    bounded = None
    for s in range(args.warmup + args.steps):
        if w.n >= 1024:  # one check of such a row can outlast the budget
            bounded = cpu_baseline_bounded(w, args.ref_seconds, cores)
            if s >= args.warmup:
                per_step.append(args.ref_seconds)
                per_checks.append(bounded['value'] * args.ref_seconds)
            continue
        t0 = time.perf_counter()
        done = 0
        while True:
            b, j = divmod(nxt % (w.B * w.k), w.k)
            O.validate_batch(w.x[b:b + 1], w.pos[b:b + 1, j:j + 1], w.cand[b:b + 1, j:j + 1], nthreads=cores)
            nxt += 1
            done += w.K
            if time.perf_counter() - t0 >= args.ref_seconds:
                break
        if s >= args.warmup:
            per_step.append(time.perf_counter() - t0)
            per_checks.append(done)
    v = float(np.sum(per_checks)) / float(np.sum(per_step))
    sample = ('proposed positions in batch order, all %d candidates of one per oracle validate_batch call on %d '
              'threads, for %.0f s per step (%d checks in the timed steps)' % (w.K, cores, args.ref_seconds,
                                                                              int(np.sum(per_checks))))
    if bounded is not None:
        sample = 'per step: ' + bounded['sample']
    line = {'impl': 'reference', 'metric': 'candidate validity checks/sec', 'value': v, 'unit': 'checks/s',
            'n_gpus': 1, 'steps': args.steps, 'warmup': args.warmup,
            'ms_per_step': float(np.mean(per_step)) * 1e3, 'higher_is_better': True, 'scaling': 'weak',
            'vs_baseline': None, 'dtype': 'int32', 'data': 'synthetic',
            'config': {'workload': args.workload, 'batch': w.B, 'seq_len': w.n, 'k': w.k, 'K': w.K,
                       'vocab': len(w.vocab), 'l2': 'n/a (host cores)', 'parallelism': 'single'},
            'cpu_baseline': {'value': v, 'unit': 'checks/s', 'cores': cores, 'kind': 'oracle', 'sample': sample},
            'e2e': {'value': v, 'unit': 'checks/s', 'h2d_bytes_per_step': 0, 'd2h_bytes_per_step': 0}}
    if bounded is not None and bounded.get('bound'):
        line['cpu_baseline']['bound'] = 'upper'
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.impl == 'reference':
        return run_reference(args)
    import torch
    import torch.distributed as dist
    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group('nccl')
    torch.cuda.set_device(local)
    dev = torch.device('cuda', local)
    import paper_2606_00722_gb300 as epic
    epic.build()
    from synth import make_workload
    w = make_workload(args.workload, args.seed + rank, k=args.k, batch=args.batch)
    g = epic.Grammar(w.grammar)
    torch.cuda.synchronize()
    tb0 = time.perf_counter()
    t = epic.LexTable(g, w.vocab, lazy_capacity=args.lazy_lex)
    table_ms = (time.perf_counter() - tb0) * 1e3  # the build synchronizes
    x0 = torch.from_numpy(w.x).to(dev)
    x = x0.clone()
    pos = torch.from_numpy(w.pos).to(dev)
    cand = torch.from_numpy(w.cand).to(dev)
    conf3 = torch.from_numpy(w.conf).to(dev)
    valid = torch.empty(w.cand.shape, dtype=torch.uint8, device=dev)
    tok = torch.empty(w.pos.shape, dtype=torch.int32, device=dev)
    conf = torch.empty(w.pos.shape, dtype=torch.float32, device=dev)
    sel = torch.empty(w.pos.shape, dtype=torch.uint8, device=dev)
    filled = torch.empty(w.pos.shape, dtype=torch.int32, device=dev)
    n_target = torch.full((w.B,), w.k, dtype=torch.int32, device=dev)  # n_t: commit every proposed position
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # > 129 MB L2
    stream = torch.cuda.current_stream()
    checks = w.B * w.k * w.K

    def step(xbuf):
        epic.validate_batch(g, t, xbuf, pos, cand, valid)
        epic.pick_candidates(cand, conf3, valid, tok, conf)
        epic.select_compatible_subset(g, t, xbuf, pos, tok, conf, sel)
        epic.commit(xbuf, pos, tok, sel)
        epic.fallback_commit(g, t, xbuf, pos, cand, conf3, n_target, sel, filled, valid=valid)

    for _ in range(args.warmup):
        x.copy_(x0)
        step(x)
    torch.cuda.synchronize()
    st_warm = t.stats(reset=True)  # the warm-up steps, from a cold lexing memo
    # ---- device-timed region: per-step events, L2 flushed before each step
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    kern = {}  # kernel -> per-step ms (CUDA events around each launch, on this stream)
    with Clocks(local) as clk:
        for i in range(args.steps):
            x.copy_(x0)
            flush.fill_(i & 255)
            ev[i][0].record(stream)
            epic.validate_batch(g, t, x, pos, cand, valid)
            ev[i][1].record(stream)
            epic.pick_candidates(cand, conf3, valid, tok, conf)
            epic.select_compatible_subset(g, t, x, pos, tok, conf, sel)
            epic.commit(x, pos, tok, sel)
            epic.fallback_commit(g, t, x, pos, cand, conf3, n_target, sel, filled, valid=valid)
            ev[i][2].record(stream)
            for kname, kms in t.kernel_times().items():  # waits for this step's kernels
                kern.setdefault(kname, []).append(kms)
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    step_ms = [a.elapsed_time(c) for a, b, c in ev]
    val_ms = [a.elapsed_time(b) for a, b, c in ev]
    st = t.stats()
    region = st['region_checks'] > 0
    # kernels of the timed region: validate's own (one walk kernel, or the
    # forward chart, good masks and region checks) + pick + two selection
    # kernels + commit + the fallback's setup and two kernels per round
    launches = st['validate_kernels'] + 5 * args.steps + 2 * st['fallback_rounds']
    sel_h = sel.cpu().numpy()
    fill_h = filled.cpu().numpy()
    commit_sizes = {'selected_per_seq': float((sel_h == 1).sum()) / w.B,
                    'fallback_per_seq': float((fill_h >= 0).sum()) / w.B,
                    'selection_overflow': int((sel_h == 2).sum())}
    ms = float(np.mean(step_ms))
    vms = float(np.mean(val_ms))
    if world > 1:
        ms, vms = max_over_ranks([ms, vms], dev)
    total_checks = checks * world
    value = job_value(checks, world, ms)
    # ---- end to end through the public API with host buffers
    hx = torch.from_numpy(w.x).pin_memory()
    hpos = torch.from_numpy(w.pos).pin_memory()
    hcand = torch.from_numpy(w.cand).pin_memory()
    hconf = torch.from_numpy(w.conf).pin_memory()
    hvalid = torch.empty(w.cand.shape, dtype=torch.uint8).pin_memory()
    hsel = torch.empty(w.pos.shape, dtype=torch.uint8).pin_memory()
    hxo = torch.empty(w.x.shape, dtype=torch.int32).pin_memory()
    hnt = torch.full((w.B,), w.k, dtype=torch.int32).pin_memory()
    hfill = torch.empty(w.pos.shape, dtype=torch.int32).pin_memory()
    e2e_ms = []
    for i in range(min(args.steps, 3)):  # the same steps end to end (at most three: long steps)
        flush.fill_(i & 255)
        a, c = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        x.copy_(hx, non_blocking=True)
        pos.copy_(hpos, non_blocking=True)
        cand.copy_(hcand, non_blocking=True)
        conf3.copy_(hconf, non_blocking=True)
        n_target.copy_(hnt, non_blocking=True)
        step(x)
        hvalid.copy_(valid, non_blocking=True)
        hsel.copy_(sel, non_blocking=True)
        hfill.copy_(filled, non_blocking=True)
        hxo.copy_(x, non_blocking=True)
        c.record(stream)
        torch.cuda.synchronize()
        e2e_ms.append(a.elapsed_time(c))
    e2e_step = float(np.mean(e2e_ms))
    h2d = w.x.nbytes + w.pos.nbytes + w.cand.nbytes + w.conf.nbytes + hnt.numel() * 4
    d2h = w.cand.size + w.pos.size + w.pos.size * 4 + w.x.nbytes
    # ---- roofline of the dominant kernel of epic_validate_batch: bit-parallel
    # Earley word operations, 3 passes (predict, scan, complete) over every
    # (node, origin) pair of the chart the kernel builds, ceil(D / 32) words
    # each, with the pairs counted by the oracle (tests/golden/census_*.json)
    # and the kernel's own launch time from CUDA events on this stream
    kms = {kname: float(np.mean(v)) for kname, v in kern.items()}
    vkern = {kname: v for kname, v in kms.items() if not kname.startswith('k_select')}
    dom = max(vkern, key=vkern.get) if vkern else None
    cen = census(args.workload, w.B)
    peak_ops, peak_ms = epic.measure_int_peak()
    peak_t = peak_ops / 1e12
    work = None
    if cen and dom in ('k_forward_gs', 'k_forward', 'k_good') and 'forward_pairs' in cen:
        work = 3.0 * cen['forward_pairs'] * cen['words']
        work_note = 'forward charts of x: %.0f (node, origin) pairs x %d words x 3 (oracle census, %s)' % (
            cen['forward_pairs'], cen['words'], cen['forward_sample'])
    elif cen and dom == 'k_validate_warp' and 'checks_pairs' in cen:
        work = 3.0 * cen['checks_pairs'] * cen['words']
        work_note = 'charts of every check: %.0f (node, origin) pairs x %d words x 3 (oracle census)' % (
            cen['checks_pairs'], cen['words'])
    else:
        work_note = 'no oracle census for %s on this workload' % dom
    achieved = (work / (kms[dom] / 1e3) / 1e12) if (work and dom) else None
    traffic = recorded_traffic(dom, args.workload) if dom else None
    # the same figure for every validate kernel whose work the census counts
    by_kernel = {}
    if cen and 'forward_pairs' in cen:
        fwork = 3.0 * cen['forward_pairs'] * cen['words']
        for kname in ('k_forward_gs', 'k_forward', 'k_good'):
            if kname in kms and kms[kname] > 0:
                a_t = fwork / (kms[kname] / 1e3) / 1e12
                by_kernel[kname] = {'achieved': a_t, 'frac': a_t / peak_t, 'kernel_ms': kms[kname]}
    roof = {'bound': 'alu', 'achieved': achieved, 'peak': peak_t, 'unit': 'T word-ops/s',
            'frac': (achieved / peak_t) if achieved else None, 'traffic': traffic,
            'peak_source': 'measured live: LOP3 + SHF microbenchmark (epic_measure_int_peak, %.2f ms)' % peak_ms,
            'kernel': dom, 'kernel_ms': kms.get(dom), 'work': work_note,
            'kernel_share_of_step': (kms[dom] / ms) if dom else None,
            'kernels_ms': {kname: round(v, 3) for kname, v in kms.items()},
            'census_kernels': by_kernel}
    line = {'metric': 'candidate validity checks/sec', 'value': value, 'unit': 'checks/s',
            'n_gpus': world, 'steps': args.steps, 'warmup': args.warmup, 'ms_per_step': ms,
            'higher_is_better': True, 'scaling': 'weak', 'vs_baseline': None, 'dtype': 'int32',
            'data': 'synthetic',
            'config': {'workload': args.workload, 'batch': w.B, 'seq_len': w.n, 'k': w.k, 'K': w.K,
                       'vocab': len(w.vocab), 'l2': 'flushed: 256 MiB write before every step',
                       'parallelism': 'replicas' if world > 1 else 'single'},
            'step': 'validate, pick, select (Alg. 4), commit, rejection fallback (Alg. 1) with n_t = k',
            'workload_note': ('clike-512 is the default: the largest configuration whose bench run fits minutes '
                              '(random-stress-1024 took 125 s per step at 8 of its 64 rows)')
            if args.workload == 'clike-512' else None,
            'step_latency_us': ms * 1e3, 'validate_checks_per_s': total_checks / (vms / 1e3),
            'valid_fraction': st['valid'] / max(1, st['checks']), 'overflow': st['overflow'],
            'gpu_launches': int(launches), 'validate_path': 'region' if region else 'walk',
            'commits': commit_sizes,
            'lex_table': {'kind': 'lazy memo (Alg. 2), %d entries' % args.lazy_lex if args.lazy_lex else 'dense',
                          'build_ms': table_ms,
                          'memo_hit_rate_warmup': ((1.0 - st_warm['lex_misses'] / st_warm['lex_lookups'])
                                                   if st_warm['lex_lookups'] else None),
                          'memo_hit_rate_timed': (1.0 - st['lex_misses'] / st['lex_lookups']) if st['lex_lookups'] else None,
                          'lookups_per_step': st['lex_lookups'] / max(1, args.steps)},
            'e2e': {'value': total_checks / (e2e_step / 1e3), 'unit': 'checks/s', 'h2d_bytes_per_step': int(h2d),
                    'd2h_bytes_per_step': int(d2h)},
            'roofline': roof, 'clocks': clk.summary()}
    if rank == 0:
        if world == 1 and not args.no_cpu_baseline:
            line['cpu_baseline'] = cpu_baseline(w, args.cpu_seconds)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def max_over_ranks(values, device=None):
    """Element-wise maximum over all ranks of the default process group (the
    job's time is its slowest rank's)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor(values, dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


def job_value(checks_per_rank, world, ms):
    """Whole-job throughput: the checks all ranks processed over the slowest
    rank's step time."""
    return checks_per_rank * world / (ms / 1e3)


if __name__ == '__main__':
    main()

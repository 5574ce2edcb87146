"""Host-side arithmetic of bench.py's roofline line (CPU): the oracle census
it takes the algorithmic work from, and the recorded DRAM traffic it reads
only while the kernel's sources are the ones the counters were taken on."""
import json
import os

import pytest

import bench


def test_census_scales_the_sample_mean_to_the_batch():
    here = os.path.dirname(os.path.abspath(__file__))
    for name in ('clike-512', 'random-stress-1024', 'json-schema'):
        path = os.path.join(here, 'golden', 'census_%s.json' % name)
        if not os.path.exists(path):
            continue
        with open(path) as f:
            d = json.load(f)
        per = [r['pairs'] for r in d['per_seq']]
        c = bench.census(name, d['batch'])
        assert c['words'] == (d['D'] + 31) // 32
        assert c['forward_pairs'] == pytest.approx(sum(per) / len(per) * d['batch'])


def test_census_of_an_unknown_workload_is_none():
    assert bench.census('no-such-workload', 4) is None


def test_recorded_traffic_needs_matching_sources(tmp_path, monkeypatch):
    (tmp_path / 'profiles').mkdir()
    (tmp_path / 'profiles' / 'traffic_k_good_w.txt').write_text(
        '# comment: ignored\nkernel: k_good\nsource_sha16: abc\ndram_bytes_per_launch: 1234.5\n')
    monkeypatch.setattr(bench, 'ROOT', str(tmp_path))
    monkeypatch.setattr(bench, 'kernel_sha', lambda k: 'abc')
    assert bench.recorded_traffic('k_good', 'w') == 1234.5
    monkeypatch.setattr(bench, 'kernel_sha', lambda k: 'changed')
    assert bench.recorded_traffic('k_good', 'w') is None
    assert bench.recorded_traffic('k_check', 'w') is None


def test_committed_traffic_records_are_well_formed():
    here = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    prof = os.path.join(here, 'profiles')
    for fn in os.listdir(prof):
        if not fn.startswith('traffic_'):
            continue
        rec = {}
        with open(os.path.join(prof, fn)) as f:
            for line in f:
                if ':' in line and not line.startswith('#'):
                    k, v = line.split(':', 1)
                    rec[k.strip()] = v.strip()
        assert fn == 'traffic_%s_%s.txt' % (rec['kernel'], rec['workload'])
        assert rec['kernel'] in bench.KERNEL_SOURCES
        assert len(rec['source_sha16']) == 16
        assert float(rec['dram_bytes_per_launch']) > 0

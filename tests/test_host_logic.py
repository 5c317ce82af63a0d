"""Host-side logic without a GPU: the key that ties a measured instruction count
to the simulator's code, and the sweep helpers' arithmetic."""
import importlib.util
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


def test_strip_comments_keeps_code_and_literals():
    b = _bench()
    src = 'int a = 1; // note\n/* block\n comment */ const char* s = "// kept /* too */";\nchar c = \'/\';\n'
    out = b._strip_comments(src)
    assert "note" not in out and "block" not in out
    assert '"// kept /* too */"' in out and "'/'" in out and "int a = 1;" in out


def test_source_key_ignores_comments_but_not_code(tmp_path, monkeypatch):
    b = _bench()
    base = b._source_hash()
    files = {}
    for rel in b.SIM_SOURCES:
        dst = tmp_path / rel
        dst.parent.mkdir(parents=True, exist_ok=True)
        dst.write_text(open(os.path.join(ROOT, rel), encoding="utf-8").read())
        files[rel] = dst
    monkeypatch.setattr(b, "ROOT", str(tmp_path))
    assert b._source_hash() == base
    sim = files[b.SIM_SOURCES[0]]
    sim.write_text("// a new comment\n" + sim.read_text())
    assert b._source_hash() == base
    sim.write_text(sim.read_text().replace("kRecipN = 1024", "kRecipN = 512"))
    assert b._source_hash() != base


def test_sweep_arithmetic():
    pytest.importorskip("torch")
    from paper_2609_16206_gb300 import sweep
    from paper_2609_16206_gb300 import workloads as W
    # contiguous near-equal split covering every replica once
    for total, world in ((10, 3), (4096, 8), (5, 8)):
        parts = [sweep.shard_split(total, world, r) for r in range(world)]
        assert sum(c for _, c in parts) == total
        assert all(parts[r][0] + parts[r][1] == parts[r + 1][0] for r in range(world - 1))
        assert max(c for _, c in parts) - min(c for _, c in parts) <= 1
    assert sweep.load_rate(3000, 29 / 30) == 2900 and sweep.load_rate(1, 0.1) == 1
    assert len(sweep.calibration_sweep_cfgs()) == 5 * 4 * 4
    assert len(W.mispriced_sets()) == 65 and sweep.NOISE_SIGMAS[0] == 0.0 and sweep.NOISE_SIGMAS[-1] == 1.5

"""Pins of the oracle's Philox4x32-10 and probe mapping (CPU only)."""
import os

import numpy as np
import pytest

import philox_ref

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat():
    rows = []
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        w = [int(x, 16) for x in line.split()]
        rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


def test_philox_known_answers(oracle_mod):
    rows = _kat()
    assert len(rows) == 3
    for ctr, key, want in rows:
        got = oracle_mod.philox4x32_10(ctr, key)
        assert [int(x) for x in got] == want


@pytest.mark.skipif(not philox_ref.available(), reason="torch Philox header not found")
def test_philox_matches_torch_engine(oracle_mod):
    rng = np.random.default_rng(7)
    seeds = [0, 1, 0xDEADBEEFCAFEF00D, int(rng.integers(0, 2**63))]
    for seed in seeds:
        ctrs = rng.integers(0, 2**32, size=(16, 4), dtype=np.uint64)
        ctrs[0] = 0
        ref = philox_ref.blocks(seed, ctrs)
        key = (seed & 0xFFFFFFFF, seed >> 32)
        for c, r in zip(ctrs, ref):
            assert (oracle_mod.philox4x32_10(c, key) == r).all()


@pytest.mark.skipif(not philox_ref.available(), reason="torch Philox header not found")
@pytest.mark.parametrize("seed,step,expert,probe,p0,count", [
    (0, 0, 0, 0, 0, 300),
    (0, 5, 3, 17, 4000, 700),
    (123456789012, 2**32 + 9, 255, 1023, 8_300_000, 260),
])
def test_probe_mapping_matches_torch_engine(oracle_mod, seed, step, expert, probe, p0, count):
    want = philox_ref.rademacher(seed, step, expert, probe, p0, count)
    got = oracle_mod.rademacher(seed, step, expert, probe, p0, count)
    assert got.dtype == np.int8
    assert (got == want).all()


def test_probe_statistics(oracle_mod):
    # dense Rademacher: E[z] = 0, E[z_a z_b] = 0 (a != b), z in {-1, +1}
    z = oracle_mod.rademacher(0, 0, 0, 0, 0, 1 << 20).astype(np.float64)
    assert set(np.unique(z)) == {-1.0, 1.0}
    assert abs(z.mean()) < 5 / np.sqrt(z.size)
    assert abs((z[:-1] * z[1:]).mean()) < 5 / np.sqrt(z.size)
    z2 = oracle_mod.rademacher(0, 0, 0, 1, 0, 1 << 20).astype(np.float64)
    assert abs((z * z2).mean()) < 5 / np.sqrt(z.size)
    z3 = oracle_mod.rademacher(0, 0, 1, 0, 0, 1 << 20).astype(np.float64)
    assert abs((z * z3).mean()) < 5 / np.sqrt(z.size)
    z4 = oracle_mod.rademacher(0, 1, 0, 0, 0, 1 << 20).astype(np.float64)
    assert abs((z * z4).mean()) < 5 / np.sqrt(z.size)

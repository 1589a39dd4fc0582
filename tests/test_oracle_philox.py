"""Pins for the oracle's random-number layer (Philox4x32-10, uniforms, Box-Muller, SplitMix64)."""
import os
import subprocess

import numpy as np
import pytest
from scipy import stats

from oracle import philox

HERE = os.path.dirname(os.path.abspath(__file__))


def _read_golden(name):
    rows = []
    with open(os.path.join(HERE, "golden", name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append([int(t, 16) for t in line.split()])
    return rows


def test_philox_known_answer_vectors():
    for row in _read_golden("philox4x32_10_kat.txt"):
        c0, c1, c2, c3, k0, k1 = row[:6]
        out = philox.philox4x32_10(c0, c1, c2, c3, k0, k1)
        assert [int(v) for v in out] == row[6:]


def test_philox_matches_torch_source_engine(tmp_path):
    """Run PyTorch's source-level Philox engine header on random counters and compare words."""
    torch = pytest.importorskip("torch")
    inc = os.path.join(os.path.dirname(torch.__file__), "include")
    exe = str(tmp_path / "philox_check")
    r = subprocess.run(["g++", "-std=c++17", "-O1", "-I" + inc,
                        os.path.join(HERE, "philox_torch_check.cpp"), "-o", exe],
                       capture_output=True, text=True)
    if r.returncode != 0:
        pytest.skip("cannot build the torch header check: " + r.stderr[-200:])
    rng = np.random.Generator(np.random.PCG64(7))
    words = rng.integers(0, 2 ** 32, size=(64, 6), dtype=np.uint64)
    lines = []
    for c0, c1, c2, c3, k0, k1 in words:
        seed = int(k1) << 32 | int(k0)
        subseq = int(c3) << 32 | int(c2)
        offset = int(c1) << 32 | int(c0)
        lines.append("%d %d %d" % (seed, subseq, offset))
    out = subprocess.run([exe], input="\n".join(lines) + "\n", capture_output=True,
                         text=True, check=True).stdout.split("\n")
    for (c0, c1, c2, c3, k0, k1), line in zip(words, out):
        mine = philox.philox4x32_10(c0, c1, c2, c3, k0, k1)
        assert ["%08x" % int(v) for v in mine] == line.split()


def test_splitmix64_published_outputs():
    expect = [row[0] for row in _read_golden("splitmix64.txt")]
    assert [philox.round_seed(0, r) for r in range(3)] == expect


def test_uniform_is_open_interval_and_exact():
    assert philox.uniform_of(0) == 2.0 ** -33
    assert philox.uniform_of(2 ** 32 - 1) == 1.0 - 2.0 ** -33
    assert 0.0 < philox.uniform_of(0) < philox.uniform_of(2 ** 32 - 1) < 1.0


def test_streams_are_uniform_and_distinct():
    b = np.arange(20000)
    eta = philox.coins(123, b, 4)
    assert eta.shape == (20000, 4)
    assert stats.kstest(eta.ravel(), "uniform").pvalue > 1e-3
    w = philox.usample_uniform(123, b)
    assert stats.kstest(w, "uniform").pvalue > 1e-3
    # distinct streams / steps / seeds give (essentially) uncorrelated values
    assert abs(np.corrcoef(eta[:, 0], w)[0, 1]) < 0.03
    assert abs(np.corrcoef(eta[:, 0], eta[:, 1])[0, 1]) < 0.03
    assert abs(np.corrcoef(eta[:, 0], philox.coins(124, b, 1)[:, 0])[0, 1]) < 0.03


def test_box_muller_normals():
    z = philox.normals(5, np.arange(64), 4099, philox.STREAM_RESID)
    assert z.shape == (64, 4099)
    flat = z.ravel()
    assert abs(flat.mean()) < 5 * 1 / np.sqrt(flat.size)
    assert abs(flat.var() - 1.0) < 5 * np.sqrt(2.0 / flat.size)
    assert stats.kstest(flat, "norm").pvalue > 1e-3
    # element i comes from counter block i // 4: a prefix does not depend on d
    z_short = philox.normals(5, 3, 10, philox.STREAM_RESID)
    np.testing.assert_array_equal(z_short, z[3, :10])
    # the pair (w0, w1) gives (r cos, r sin): z0^2 + z1^2 = -2 ln u0
    w = philox.philox4x32_10(3, 0, philox.STREAM_RESID, 0, *philox.key_of(5))
    r2 = -2.0 * np.log(philox.uniform_of(w[0]))
    assert np.isclose(z[3, 0] ** 2 + z[3, 1] ** 2, r2, rtol=1e-13)


def test_round_seeds_differ():
    seeds = {philox.round_seed(42, r) for r in range(1000)}
    assert len(seeds) == 1000

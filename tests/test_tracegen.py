"""The seeded input generator: determinism, shapes and value ranges of the five workloads."""
import json
import math
import os

import numpy as np
import pytest

import tracegen as tg

SUMMARIES = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "config_summaries.json")))


@pytest.mark.parametrize("k", range(5))
def test_digest_matches_committed(k):
    assert tg.digest(tg.config(k)) == SUMMARIES["configs"][k]["sha256"]


def test_exp2_series():
    lib = tg._load()
    for x in np.linspace(0, 26, 1000):
        assert math.isclose(lib.tg_debug_exp2(float(x)), 2.0 ** float(x), rel_tol=1e-14)


def test_uniform_int_range_and_spread():
    lib = tg._load()
    vals = [lib.tg_debug_uniform_int(3, 5, 9, k) for k in range(3000)]
    assert set(vals) == {5, 6, 7, 8, 9}
    counts = np.bincount(np.array(vals) - 5)
    assert counts.min() > 500  # expected 600 each


def test_determinism():
    a = tg.random_batch(42, 3, 50, 60)
    b = tg.random_batch(42, 3, 50, 60)
    assert tg.digest(a) == tg.digest(b)
    c = tg.random_batch(43, 3, 50, 60)
    assert tg.digest(a) != tg.digest(c)


def _common_checks(ts):
    assert ts.trace_ptr[0] == 0 and ts.trace_ptr[-1] == ts.n_tensors
    assert (np.diff(ts.trace_ptr) >= 0).all()
    for b in range(ts.n_traces):
        T, a, f, s = ts.trace(b)
        assert (a >= 0).all() and (f > a).all() and (f <= T).all() and (s > 0).all()


def test_random_workloads_shape():
    for k, (B, n, T) in ((0, (1, 64, 128)), (2, (4096, 512, 1024))):
        ts = tg.config(k)
        assert (ts.n_traces, ts.max_tensors, ts.max_steps) == (B, n, T)
        _common_checks(ts)
        assert (ts.size_bytes % 64 == 0).all()
        assert ts.size_bytes.min() >= 64 and ts.size_bytes.max() <= 1 << 20
        life = ts.free_step - ts.alloc_step
        assert abs(life.mean() - 2.0) < 0.05 or k == 0  # 1 + Geometric(0.5) has mean 2


def test_resnet_chain():
    ts = tg.config(1)
    assert ts.n_tensors == 374 and ts.steps.tolist() == [160]
    _common_checks(ts)
    shapes = {4 * c * h * h for c, h in ((64, 112), (256, 56), (512, 28), (1024, 14), (2048, 7))}
    assert set(ts.size_bytes.tolist()) <= shapes
    life = ts.free_step - ts.alloc_step
    assert life.max() <= 4


def test_long_tail():
    ts = tg.config(3)
    assert ts.n_tensors == 20000 and ts.steps.tolist() == [10000]
    _common_checks(ts)
    life = ts.free_step - ts.alloc_step
    long_ = life >= 100  # short lifetimes reach 100 with probability 0.6^99
    assert 900 <= long_.sum() <= 1000
    assert (ts.size_bytes % 64 == 0).all() and ts.size_bytes.max() <= 64 << 20


def test_seq2seq():
    ts = tg.config(4)
    assert ts.n_traces == 256 and ts.max_tensors == 2000 and ts.max_steps == 4000
    _common_checks(ts)
    for b in range(0, 256, 17):
        T, a, f, s = ts.trace(b)
        full = (a == 0) & (f == T)
        assert full.sum() == 40
        per_token = np.unique(s)
        assert len(per_token) <= 4  # {4BSH, 4BH} x H in {1024, 4096}

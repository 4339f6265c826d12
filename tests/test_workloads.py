"""Recipes of the seeded synthetic workloads (no GPU needed)."""
import numpy as np
import pytest

from paper_2603_02565_gb300 import workloads as wl


def test_round_to_bf16_is_nearest_even():
    x = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 1e-30, 3.0e38], dtype=np.float32)
    r = wl.round_to_bf16(x)
    # 1 + 2^-8 is halfway between 1 and 1 + 2^-7: ties to the even mantissa (1.0)
    assert r[0] == 1.0 and r[1] == 1.0 and r[2] == np.float32(1.0 + 2 ** -6)
    assert r[3] == -2.5
    assert (wl.round_to_bf16(r) == r).all()
    assert (r.view(np.uint32) & 0xFFFF == 0).all()


def test_sequences_have_distinct_items_and_valid_range():
    rng = np.random.default_rng(0)
    for zipf in (None, 1.1, 1.3):
        c = wl.sample_sequences(rng, 8, 30, 20, 6, zipf)
        assert c.shape == (8, 20, 6) and c.dtype == np.int32
        assert c.min() >= 0 and c.max() < 30
        for row in c.reshape(-1, 6):
            assert len(set(row.tolist())) == 6


def test_zipf_popularity_is_skewed():
    rng = np.random.default_rng(1)
    c = wl.sample_sequences(rng, 1, 100, 4000, 1, 1.1)
    counts = np.bincount(c.ravel(), minlength=100)
    top = np.sort(counts)[::-1]
    # rank 1 has weight 1 / H, H = sum r^-1.1 (~ 4.4 for 100 ranks)
    H = (np.arange(1, 101) ** -1.1).sum()
    assert abs(top[0] / 4000 - 1 / H) < 0.03


def test_workloads_are_deterministic_and_bf16_valued():
    a = wl.make_workload("serving", B=4)
    b = wl.make_workload("serving", B=4)
    assert (a.cand_idx == b.cand_idx).all() and (a.context == b.context).all()
    for arr in [a.context, a.pool, *a.weights.values()]:
        assert (wl.round_to_bf16(arr) == arr).all()
    t = wl.make_workload("tiny")
    assert t.shape == (1, 16, 20, 4, 5) and not t.cfg.io_bf16


@pytest.mark.parametrize("name,kw,U_lo,U_hi", [
    ("serving", dict(B=64), 60, 82),
    ("ksweep", dict(K=10), 65, 90),
    ("ksweep", dict(K=100), 190, 200),
])
def test_distinct_counts_match_recipe(name, kw, U_lo, U_hi):
    w = wl.make_workload(name, **kw)
    U = np.array([len(np.unique(c)) for c in w.cand_idx])
    assert U_lo <= U.mean() <= U_hi


def test_summarisation_recipe():
    w = wl.summarisation(B=3, C=8, d=16, H=2, K=16, L=64, vocab=4096)
    B, C, M, K, L = w.shape
    assert (B, C, K, L) == (3, 8, 16, 64)
    for b in range(B):
        used = np.unique(w.cand_idx[b])
        assert used[0] == 0 and used[-1] == len(used) - 1   # pool = distinct tokens, in order
        assert (w.pool[b, len(used):] == 0).all()
    # every hypothesis shares ~70% of its positions with the most common token per column
    agree = []
    for b in range(B):
        h = w.cand_idx[b]
        mode = np.array([np.bincount(col).argmax() for col in h.T])
        agree.append((h == mode).mean())
    assert 0.6 < np.mean(agree) < 0.8

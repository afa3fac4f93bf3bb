"""Pins for the oracle's model of asynchronous cache reuse across batches
(Section 3.3, "Dynamic Fusion and Reuse Mechanism" (II))."""
import numpy as np

import oracle


def test_cache_reuse_model():
    """Cross-batch reuse (Section 3.3 (II)): a row hits iff an equal row was
    executed in an earlier batch — never within its own batch."""
    a, b, c = (np.full((1, 4), v, np.int32) for v in (1, 2, 3))
    batches = [np.concatenate([a, b]), np.concatenate([b, c]), np.concatenate([c, a, b]),
               np.zeros((0, 4), np.int32)]
    hits = oracle.cache_reuse(batches)
    assert [h.tolist() for h in hits] == [[False, False], [True, False], [True, True, True], []]


def test_cache_reuse_counts_distinct_rows_once():
    rng = np.random.default_rng(0)
    pool = rng.integers(0, 1 << 30, size=(50, 8)).astype(np.int32)
    batches = [np.unique(pool[rng.integers(0, 50, 30)], axis=0) for _ in range(6)]
    hits = oracle.cache_reuse(batches)
    misses = sum(int((~h).sum()) for h in hits)
    distinct = len({r.tobytes() for b in batches for r in b})
    assert misses == distinct                 # every distinct row executes exactly once

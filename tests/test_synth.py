"""The seeded generator: determinism, exact planted duplicate counts, shapes
and the distributions the workload shapes ask for."""
import numpy as np

import synth
from synth import configs


def test_deterministic_and_seed_sensitive():
    a = synth.unit_rows(10, 64, seed=3)
    b = synth.unit_rows(10, 64, seed=3)
    c = synth.unit_rows(10, 64, seed=4)
    assert (a == b).all() and not (a == c).all()


def test_slices_agree_with_whole():
    whole = synth.unit_rows(50, 32, seed=9)
    part = synth.unit_rows(20, 32, seed=9, counter0=30)
    assert (whole[30:] == part).all()


def test_unit_norm_within_bf16_rounding():
    x = synth.unit_rows(200, 768, seed=1)
    f = (x.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    assert np.abs(np.linalg.norm(f, axis=1) - 1).max() < 4e-3


def test_gaussian_moments():
    z = np.array([synth._load().synth_normal(5, 1, i) for i in range(20000)])
    assert abs(z.mean()) < 0.03 and abs(z.std() - 1) < 0.03


def test_copy_counts_and_cross_workflow_sources():
    n, block = 4096, 64
    root = synth.copy_plan(n, int(round(0.4 * n)), seed=2, block=block)
    copies = np.nonzero(root != np.arange(n))[0]
    assert len(copies) == int(round(0.4 * n))
    assert (root[copies] // block < copies // block).all()      # earlier workflow
    assert (root[root] == root).all()                           # roots are originals


def test_token_rows_distinct_and_padded():
    lens = synth.uniform_ints(300, 64, 512, seed=0)
    assert lens.min() >= 64 and lens.max() <= 512
    t = synth.token_rows(300, 512, seed=0, lens=lens)
    assert t.min() >= 0 and t.max() < synth.VOCAB
    for i in range(300):
        assert (t[i, lens[i]:] == 0).all()
    assert len({(int(r[0]), int(r[1])) for r in t}) == 300


def test_zipf_head_frequency():
    pool, s, n = 1000, 1.1, 200000
    r = synth.zipf_ranks(n, pool, s, seed=1)
    H = (np.arange(1, pool + 1, dtype=np.float64) ** -s).sum()
    f0 = (r == 0).mean()
    assert abs(f0 - 1 / H) < 0.01
    assert np.bincount(r, minlength=pool)[:5].tolist() == sorted(
        np.bincount(r, minlength=pool)[:5].tolist(), reverse=True)


def test_config_shapes_small():
    w = configs.build_retrieval_mix(configs.TINY)
    assert w["tokens"].shape == (256, 128) and w["queries"].shape == (32, 384)
    assert w["corpus"].shape == (4096, 384)
    b = configs.build_sweep_batch(64)
    assert b["queries"].shape == (64, 768)
    assert (b["query_root"] != np.arange(64)).sum() == 13

"""Host-side arithmetic of bench.py: the algorithmic byte counts behind the
roofline figures (checked against a hand count and against each other), the
microbenchmark's lattice generator, and the throughput formula."""
import numpy as np

import bench


def test_decode_bytes_hand_count():
    # L=1, d=2, F=4, V=3, n=2, bf16 weights; prompt 5, 3 generated tokens:
    # step 1 feeds nothing (heads only), step 2 feeds 2 tokens over 5 cached keys.
    d, F, V, L, n, wb = 2, 4, 3, 1, 2, 2
    weights = (3 * d * d + d * d + 2 * d * F) * wb + (3 * d + d + F + d + 4 * d) * 4
    heads = n * V * d * wb + n * V * 4 + 2 * d * 4
    kv_step2 = (5 + 2) * d * 2 * 2 + 2 * d * 2 * 2   # keys + values read, the fed rows' written
    assert bench._decode_bytes_total(d, F, V, L, n, wb, 5, 3) == 2 * heads + weights + kv_step2


def test_batched_bytes_reduce_to_the_single_sequence_count():
    args = (1024, 4096, 1025, 12, 4, 2)
    for prompt, gen in [(289, 750), (40, 13), (100, 1)]:
        assert bench._batched_decode_bytes([prompt], [gen], *args) == bench._decode_bytes_total(*args, prompt, gen)


def test_batched_bytes_share_weights_between_sequences():
    args = (64, 256, 33, 2, 4, 2)
    one = bench._decode_bytes_total(*args, 10, 8)
    two = bench._batched_decode_bytes([10, 10], [8, 8], *args)
    d, F, V, L, n, wb = args
    weights = L * ((3 * d * d + d * d + 2 * d * F) * wb + (3 * d + d + F + d + 4 * d) * 4)
    heads = n * V * d * wb + n * V * 4 + 2 * d * 4
    # 8 tokens at n = 4: a first step that feeds nothing (heads only), then one that feeds 4
    # tokens (heads, weights, keys and values); the second sequence adds only its keys and values
    assert two - one == one - 2 * heads - weights


def test_c5_lattices():
    ids, lp = bench.c5_lattices(300, 8, 16, 1025, seed=3)
    assert ids.shape == (300, 8, 16) and lp.shape == (300, 8, 16)
    assert ids.min() >= 0 and ids.max() < 1025
    flat = ids.reshape(-1, 16)
    assert all(len(set(r.tolist())) == 16 for r in flat)
    assert np.all(lp <= 0) and np.all(np.diff(lp, axis=2) <= 0)
    again, lp2 = bench.c5_lattices(300, 8, 16, 1025, seed=3)
    assert np.array_equal(ids, again) and np.array_equal(lp, lp2)


def test_job_tokens_per_s():
    assert bench.job_tokens_per_s(2, 3, 1.5) == 2 * 3 * bench.GEN * bench.BATCH / 1.5

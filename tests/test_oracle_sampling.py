"""Pins of the oracle's path sampling (top-k sampling over the lattice): the
counter-based generator is SplitMix64 (checked against its published first
outputs for seed 0 of the sequential generator), paths are drawn with the
exact path posterior (brute force over all k^n paths), k = 1 gives the
per-head argmax, and a dominant path is always drawn."""
import itertools

import numpy as np
import pytest

from oracle import select as S


def test_splitmix64_reference_outputs():
    # the sequential SplitMix64 generator seeded with 0 (state += golden gamma, then mix)
    # starts e220a8397b1dcdaf, 6e789e6aa1b965f4, 06c45d188009454f
    assert S.splitmix64(0) == 0xE220A8397B1DCDAF
    assert S.splitmix64(0x9E3779B97F4A7C15) == 0x6E789E6AA1B965F4
    assert S.splitmix64((2 * 0x9E3779B97F4A7C15) & ((1 << 64) - 1)) == 0x06C45D188009454F


def test_uniforms_are_in_range_and_distinct():
    u = [S.path_uniform(7, b, g, t) for b in range(3) for g in range(5) for t in range(8)]
    assert all(0.0 <= x < 1.0 for x in u)
    assert len(set(u)) == len(u)


def _posterior(ids, lp, lq):
    n, k = lp.shape
    paths, logw = [], []
    for st in itertools.product(range(k), repeat=n):
        w = lp[0, st[0]] + sum(lq[ids[t - 1, st[t - 1]], ids[t, st[t]]] + lp[t, st[t]] for t in range(1, n))
        paths.append(tuple(ids[t, st[t]] for t in range(n)))
        logw.append(w)
    logw = np.array(logw, dtype=np.float64)
    p = np.exp(logw - logw.max())
    return paths, p / p.sum()


def test_sampling_matches_the_exact_path_posterior():
    rng = np.random.default_rng(5)
    V, n, k = 12, 3, 3
    lq = np.log(rng.dirichlet(np.ones(V), size=V))
    ids = np.stack([rng.permutation(V)[:k] for _ in range(n)]).astype(np.int32)
    lp = np.log(rng.dirichlet(np.ones(k), size=n)) * 0.7
    paths, p = _posterior(ids, lp, lq)
    draws = 20000
    counts = {q: 0 for q in paths}
    for i in range(draws):
        u = [S.path_uniform(11, 0, i, t) for t in range(n)]
        counts[tuple(S.sample_path(ids, lp, lq, u)[0])] += 1
    freq = np.array([counts[q] / draws for q in paths])
    assert np.abs(freq - p).max() < 4.5 * np.sqrt(p.max() * (1 - p.max()) / draws) + 1e-3
    chi2 = ((freq - p) ** 2 / np.maximum(p, 1e-12)).sum() * draws
    assert chi2 < 26 + 3 * np.sqrt(2 * 26)   # 26 degrees of freedom


def test_k1_and_dominant_path():
    rng = np.random.default_rng(6)
    V, n = 9, 4
    lq = np.log(rng.dirichlet(np.ones(V), size=V))
    ids = rng.integers(0, V, size=(n, 1)).astype(np.int32)
    lp = np.zeros((n, 1))
    assert S.sample_path(ids, lp, lq, [0.99] * n)[0].tolist() == ids[:, 0].tolist()
    ids = np.stack([rng.permutation(V)[:4] for _ in range(n)]).astype(np.int32)
    lp = np.full((n, 4), -60.0)
    lp[:, 2] = 0.0
    for g in range(20):
        u = [S.path_uniform(3, 1, g, t) for t in range(n)]
        assert S.sample_path(ids, lp, lq, u)[0].tolist() == ids[:, 2].tolist()


def test_categorical_hand_case():
    # weights 1, 1, 2: u = 0.3 -> target 1.2 of 4 lies in [1, 2): index 1, margin 0.2 / 4
    i, m = S._categorical(np.log(np.array([1.0, 1.0, 2.0])), 0.3)
    assert i == 1 and abs(m - 0.05) < 1e-12
    i, m = S._categorical(np.array([-np.inf, 0.0, -np.inf]), 0.999)   # one positive weight: margin 1
    assert i == 1 and m == 1.0
    i, _ = S._categorical(np.array([0.0, -np.inf]), 0.999999)          # never a zero-weight index
    assert i == 0


def test_union_sampling_matches_the_exact_posterior():
    rng = np.random.default_rng(8)
    V, n, k = 10, 3, 2
    lq = np.log(rng.dirichlet(np.ones(V), size=V))
    logp = np.log(rng.dirichlet(np.ones(V) * 0.5, size=n)).astype(np.float32)
    ids = np.stack([np.argsort(-logp[t], kind="stable")[:k] for t in range(n)]).astype(np.int32)
    states = np.unique(ids)
    m = len(states)
    paths, p = _posterior(np.tile(states, (n, 1)), logp[:, states].astype(np.float64), lq)
    draws = 20000
    counts = {q: 0 for q in paths}
    for i in range(draws):
        u = [S.path_uniform(4, 2, i, t) for t in range(n)]
        counts[tuple(S.sample_path_union(ids, logp, lq, u)[0])] += 1
    freq = np.array([counts[q] / draws for q in paths])
    dof = m ** n - 1
    chi2 = ((freq - p) ** 2 / np.maximum(p, 1e-12)).sum() * draws
    assert chi2 < dof + 4 * np.sqrt(2 * dof)


def test_forced_position_is_kept():
    rng = np.random.default_rng(9)
    V, n, k = 16, 4, 5
    lq = np.log(rng.dirichlet(np.ones(V), size=V))
    ids = np.stack([rng.permutation(V)[:k] for _ in range(n)]).astype(np.int32)
    lp = np.log(rng.dirichlet(np.ones(k), size=n))
    lp[0, 1:] = -np.inf
    seen = set()
    for g in range(200):
        path, _ = S.sample_path(ids, lp, lq, [S.path_uniform(1, 0, g, t) for t in range(n)])
        assert path[0] == ids[0, 0]
        seen.add(tuple(path))
    assert len(seen) > 10   # the drafts after it still vary


def test_hand_worked_draws():
    import json
    import os
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "sampling_hand.json")))
    lq = np.log(np.array(g["log_q_probs"])).astype(np.float32)
    ids = np.array(g["cand_ids"], dtype=np.int32)
    lp = np.log(np.array(g["cand_probs"])).astype(np.float32)
    for case in g["cases"]:
        path, margin = S.sample_path(ids, lp, lq, case["uniforms"])
        assert path.tolist() == case["path"], case["note"]
        assert margin > 0.05

"""Pins of the oracle's heads, log-softmax, top-k and Viterbi (Sec. III-B, III-C).

Each pin comes from outside the oracle: brute-force enumeration, hand-worked
lattices (tests/golden/viterbi_hand.json), reductions with a known answer,
and a library sort."""
import itertools
import json
import os

import numpy as np
import pytest

import synth
from oracle import select as S

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "viterbi_hand.json")


def brute_force(cand_ids, cand_logp, log_q):
    """Every k^n path of one lattice, scored left to right: s_1 + LQ + s_2 + LQ + ..."""
    n, k = cand_ids.shape
    out = []
    for states in itertools.product(range(k), repeat=n):
        total = np.float32(cand_logp[0, states[0]])
        for t in range(1, n):
            total = np.float32(total + log_q[cand_ids[t - 1, states[t - 1]], cand_ids[t, states[t]]])
            total = np.float32(total + cand_logp[t, states[t]])
        out.append((states, total))
    return out


def random_log_q(v, seed):
    return np.log(synth.uniform(seed, "test_log_q", v * v) + 1e-3).astype(np.float32).reshape(v, v)


@pytest.mark.parametrize("n,k", [(1, 4), (2, 3), (3, 4), (4, 2), (5, 3), (6, 2), (4, 4)])
def test_viterbi_equals_brute_force(n, k):
    v = 40
    log_q = random_log_q(v, 11 + n * 7 + k)
    ids, logp = synth.make_lattice(150, n, k, v, seed=100 + 10 * n + k)
    path, state, score = S.viterbi(ids, logp, log_q)
    for b in range(ids.shape[0]):
        paths = brute_force(ids[b], logp[b], log_q)
        best = max(s for _, s in paths)
        assert score[b] == best                       # bit-exact float32
        winners = [st for st, s in paths if s == best]
        if len(winners) == 1:
            assert tuple(state[b]) == winners[0]
            assert list(path[b]) == [ids[b, t, j] for t, j in enumerate(winners[0])]


def test_viterbi_ties_reach_the_max():
    v = 12
    log_q = np.round(random_log_q(v, 5) * 2.0) / 2.0
    ids, logp = synth.make_lattice(300, 4, 3, v, seed=9, quantum=0.5)
    _, state, score = S.viterbi(ids, logp, log_q.astype(np.float32))
    for b in range(ids.shape[0]):
        paths = dict(brute_force(ids[b], logp[b], log_q.astype(np.float32)))
        assert paths[tuple(state[b])] == score[b] == max(paths.values())


def test_viterbi_golden_hand_worked():
    cases = json.load(open(GOLDEN))["cases"]
    for case in cases:
        lq = np.array(case["log_q"], dtype=np.float32)
        ids = np.array(case["cand_ids"], dtype=np.int32)[None]
        lp = np.array(case["cand_logp"], dtype=np.float32)[None]
        path, state, score = S.viterbi(ids, lp, lq)
        assert path[0].tolist() == case["path"], case["name"]
        assert state[0].tolist() == case["states"], case["name"]
        assert float(score[0]) == case["score"], case["name"]


def test_k1_is_per_head_argmax():
    v = 30
    ids, logp = synth.make_lattice(50, 6, 1, v, seed=3)
    path, _, _ = S.viterbi(ids, logp, random_log_q(v, 4))
    assert np.array_equal(path, ids[:, :, 0])


def test_uniform_q_is_per_head_argmax():
    v = 30
    ids, logp = synth.make_lattice(80, 5, 4, v, seed=5)     # rows sorted best first
    lq = np.full((v, v), np.float32(np.log(1.0 / v)), dtype=np.float32)
    path, _, _ = S.viterbi(ids, logp, lq)
    assert np.array_equal(path, ids[:, :, 0])


def test_sticky_diagonal_stays_on_shared_token():
    v, n, k = 20, 4, 3
    lq = np.full((v, v), -1e4, dtype=np.float32)
    np.fill_diagonal(lq, 0.0)
    ids = np.array([[[3, 7, 9], [5, 9, 1], [9, 2, 4], [0, 6, 9]]], dtype=np.int32)
    lp = np.array([[[-0.1, -0.2, -3.0], [-0.1, -2.0, -0.3], [-1.5, -0.1, -0.2],
                    [-0.1, -0.2, -2.5]]], dtype=np.float32)
    path, _, _ = S.viterbi(ids, lp, lq)
    assert path[0].tolist() == [9, 9, 9, 9]


def test_log_softmax_normalises_and_is_shift_invariant():
    logits = 3.0 * synth.normal(1, "ls", 4 * 1025).reshape(4, 1025)
    logp, lse = S.log_softmax(logits)
    assert np.all(np.abs(np.exp(logp).sum(axis=1) - 1.0) < 1e-5)
    logp2, lse2 = S.log_softmax(logits + 17.25)
    assert np.allclose(logp, logp2, atol=1e-12)
    assert np.allclose(lse2 - lse, 17.25, atol=1e-12)
    assert np.allclose(lse, np.log(np.exp(logits).sum(axis=1)), atol=1e-12)


@pytest.mark.parametrize("k", [1, 4, 16, 25])
def test_top_k_matches_stable_lexicographic_sort(k):
    scores = np.round(synth.normal(2, "tk", 3 * 200).reshape(3, 200) * 4) / 4   # many ties
    scores = scores.astype(np.float32)
    ids_v, vals_v = S.top_k_rows(scores, k)
    for r in range(3):
        order = np.lexsort((np.arange(200), -scores[r].astype(np.float64)))[:k]
        ids, vals = S.top_k(scores[r], k)
        assert ids.tolist() == order.tolist()
        assert ids_v[r].tolist() == order.tolist()
        assert np.array_equal(vals, scores[r][order]) and np.array_equal(vals_v[r], vals)


def test_union_lattice_brute_force_and_dominates_reading_a():
    v, n, k = 25, 3, 3
    log_q = random_log_q(v, 21)
    logits = synth.normal(22, "union", 60 * n * v).reshape(60, n, v)
    for b in range(60):
        logp32 = S.log_softmax(logits[b])[0].astype(np.float32)
        ids, vals = S.top_k_rows(logp32, k)
        path_b, score_b = S.viterbi_union(ids, logp32, log_q)
        states = np.unique(ids.reshape(-1))
        lat_ids = np.broadcast_to(states, (n, states.shape[0]))
        best = max(s for _, s in brute_force(lat_ids, logp32[:, states], log_q))
        assert score_b == best
        _, _, score_a = S.viterbi(ids[None], vals[None], log_q)
        assert score_b >= score_a[0]


def test_margin_matches_brute_force_runner_up():
    v = 15
    log_q = random_log_q(v, 31)
    ids, logp = synth.make_lattice(60, 3, 3, v, seed=32)
    margin = S.viterbi_margin(ids, logp, log_q)
    for b in range(60):
        exact = sorted((float(np.float64(logp[b, 0, st[0]]) + sum(
            float(log_q[ids[b, t - 1, st[t - 1]], ids[b, t, st[t]]]) + float(logp[b, t, st[t]])
            for t in range(1, 3))) for st, _ in brute_force(ids[b], logp[b], log_q)), reverse=True)
        assert abs(margin[b] - (exact[0] - exact[1])) < 1e-9


@pytest.mark.parametrize("path,remaining,expect", [
    ([5, 6, 7, 8], 100, (4, False)),
    ([5, 1024, 7, 8], 100, (2, True)),
    ([1024, 6, 7, 8], 100, (1, True)),
    ([5, 6, 7, 8], 3, (3, True)),
    ([5, 6, 7, 8], 4, (4, True)),
    ([5, 6, 1024, 8], 2, (2, True)),
])
def test_accept_all(path, remaining, expect):
    assert S.accept_all(np.array(path), 1024, remaining) == expect

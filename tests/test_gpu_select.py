"""GPU parity of the Viterbi selection and the heads + log-softmax + top-k kernels."""
import json
import os

import numpy as np
import pytest

import synth
from oracle import select as S

from gpu_util import assert_logits_close, lib_module, logp32, MARGIN

pytestmark = pytest.mark.gpu


def _run_viterbi(ids, lp, lq, remaining=None, eos=1024):
    import torch
    mtp = lib_module()
    b, n, k = ids.shape
    dev = torch.device("cuda")
    t_ids = torch.from_numpy(np.ascontiguousarray(ids)).to(dev)
    t_lp = torch.from_numpy(np.ascontiguousarray(lp)).to(dev)
    t_q = torch.from_numpy(np.ascontiguousarray(lq)).to(dev)
    t_rem = None if remaining is None else torch.from_numpy(remaining.astype(np.int32)).to(dev)
    path = torch.zeros((b, n), dtype=torch.int32, device=dev)
    score = torch.zeros(b, dtype=torch.float32, device=dev)
    acc = torch.zeros(b, dtype=torch.int32, device=dev)
    rb = torch.full((b,), -1, dtype=torch.int32, device=dev)
    mtp.mtp_viterbi(b, n, k, lq.shape[0], eos, t_ids, t_lp, t_q, t_rem, path, score, acc, rb,
                    torch.cuda.current_stream())
    torch.cuda.synchronize()
    return path.cpu().numpy(), score.cpu().numpy(), acc.cpu().numpy(), rb.cpu().numpy()


@pytest.mark.parametrize("n,k", [(1, 1), (1, 4), (2, 3), (4, 4), (5, 7), (8, 16), (8, 32), (3, 25)])
def test_viterbi_bit_exact(n, k):
    v = 1025
    lq = synth.transition_log_q(v)
    ids, lp = synth.make_lattice(2000, n, k, v, seed=40 + n * 33 + k)
    path, score, acc, rb = _run_viterbi(ids, lp, lq)
    ref_path, _, ref_score = S.viterbi(ids, lp, lq)
    assert np.array_equal(path, ref_path)
    assert np.array_equal(score.view(np.uint32), ref_score.view(np.uint32))
    ref_acc = np.array([S.accept_all(p, 1024, n)[0] for p in ref_path])
    assert np.array_equal(acc, ref_acc) and np.all(rb == 0)


def test_viterbi_ties_and_eos_budget():
    v = 64
    lq = np.round(synth.transition_log_q(v) * 2) / 2
    lq = lq.astype(np.float32)
    ids, lp = synth.make_lattice(3000, 6, 5, v, seed=77, quantum=0.25)
    ids[::7, 2, 0] = 63                       # EOS (id 63 here) inside paths
    rem = (np.arange(3000) % 8).astype(np.int32)
    path, score, acc, _ = _run_viterbi(ids, lp, lq, remaining=rem, eos=63)
    ref_path, _, ref_score = S.viterbi(ids, lp, lq)
    assert np.array_equal(path, ref_path)
    assert np.array_equal(score, ref_score)
    ref_acc = np.array([S.accept_all(p, 63, int(r))[0] for p, r in zip(ref_path, rem)])
    assert np.array_equal(acc, ref_acc)


def test_viterbi_golden_hand_worked():
    cases = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "viterbi_hand.json")))["cases"]
    for case in cases:
        lq = np.array(case["log_q"], dtype=np.float32)
        ids = np.array(case["cand_ids"], dtype=np.int32)[None]
        lp = np.array(case["cand_logp"], dtype=np.float32)[None]
        path, score, _, _ = _run_viterbi(ids, lp, lq, eos=lq.shape[0] + 5)
        assert path[0].tolist() == case["path"], case["name"]
        assert float(score[0]) == case["score"], case["name"]


def test_viterbi_microbench_shape():
    """10^4 lattices of 8 positions x 16 candidates over V = 1025 (head microbenchmark shape)."""
    lq = synth.transition_log_q(1025)
    ids, lp = synth.make_lattice(10000, 8, 16, 1025, seed=5)
    path, score, _, _ = _run_viterbi(ids, lp, lq)
    ref_path, _, ref_score = S.viterbi(ids, lp, lq)
    assert np.array_equal(path, ref_path) and np.array_equal(score, ref_score)


def test_viterbi_empty_batch():
    mtp = lib_module()
    mtp.mtp_viterbi(0, 4, 4, 1025, 1024, None, None, None, None, None, None, None, None)


def test_viterbi_rejects_bad_sizes():
    mtp = lib_module()
    for n, k in [(0, 4), (9, 4), (4, 0), (4, 33)]:
        with pytest.raises(mtp.MTPError):
            mtp.mtp_viterbi(1, n, k, 1025, 1024, 1, 1, 1, None, 1, None, 1, None)


@pytest.mark.parametrize("batch,n,k,dtype", [(1, 4, 4, "f32"), (7, 8, 16, "bf16"), (9, 2, 25, "f32"),
                                             (256, 8, 16, "bf16")])
def test_heads_topk_parity(batch, n, k, dtype):
    import torch
    mtp = lib_module()
    from gpu_util import decoder
    model = synth.VALLE
    dec, w = decoder(model, max_batch=1, max_ctx=128)
    try:
        h = synth.make_hidden(batch, model.d_model, seed=batch)
        dev = torch.device("cuda")
        if dtype == "bf16":
            th = torch.from_numpy(h).to(dev).to(torch.bfloat16)
            dt = 1
        else:
            th = torch.from_numpy(h).to(dev)
            dt = 0
        ids = torch.zeros((batch, n, k), dtype=torch.int32, device=dev)
        lp = torch.zeros((batch, n, k), dtype=torch.float32, device=dev)
        lg = torch.zeros((batch, n, model.codec_vocab), dtype=torch.float32, device=dev)
        lse = torch.zeros((batch, n), dtype=torch.float32, device=dev)
        mtp.mtp_heads_topk(dec.ctx, batch, th, dt, n, k, ids, lp, lg, lse)
        torch.cuda.synchronize()
        ids, lp, lg, lse = (x.cpu().numpy() for x in (ids, lp, lg, lse))
        wd = {name: np.asarray(t, np.float64) for name, t in w.items()}
        rows = range(batch) if batch <= 16 else range(0, batch, 17)
        for b in rows:
            ref = S.head_logits(h[b].astype(np.float64), wd, n, model.ln_eps)
            assert_logits_close(lg[b], ref, f"row {b}")
            _, ref_lse = S.log_softmax(ref)
            assert np.abs(lse[b] - ref_lse).max() < 2e-2
            # bit-exact top-k given the kernel's own scores
            sc = logp32(lg[b], lse[b])
            r_ids, r_vals = S.top_k_rows(sc, k)
            assert np.array_equal(ids[b], r_ids) and np.array_equal(lp[b], r_vals)
            # agreement with the oracle's own decisions where they are clear
            ref_lp32 = (ref - ref_lse[:, None]).astype(np.float32)
            o_ids, _ = S.top_k_rows(ref_lp32, k)
            gaps = S.topk_gap(ref_lp32, k)
            for i in range(n):
                if gaps[i] > MARGIN:
                    assert set(o_ids[i].tolist()) == set(ids[b, i].tolist())
    finally:
        dec.close()

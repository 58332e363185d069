"""GPU parity of the fused heads kernel (Sec. III-B: each head's logits z W_i^T + b_i,
z = LN_f(h), their log-softmax and top-k in one tensor-core pass over the head weights).

Above 8 rows mtp_heads_topk and the batched decode steps run it; option
MTP_OPT_HEADS_FUSED = 0 gives the heads GEMM + selection kernel path for comparison.
Checked: logits within the bf16 bar of the oracle, lse against the oracle, the
top-k bit-exact given the kernel's own logits and lse (ranking on logp, equal
values by id), agreement with the oracle's decisions where they are clear,
ragged tiles, every top_k bucket, outputs left out, and tie-heavy rows where
whole vocabulary slices share one score."""
import numpy as np
import pytest

import synth
from oracle import select as S

from gpu_util import assert_logits_close, decoder, lib_module, logp32, MARGIN

pytestmark = pytest.mark.gpu

OPT_HEADS_FUSED = 11


def _heads(dec, h, n, k, fused=True, want_logits=True, want_lse=True):
    import torch
    mtp = lib_module()
    mtp.mtp_set_option(dec.ctx, OPT_HEADS_FUSED, 1 if fused else 0)
    assert mtp.mtp_get_option(dec.ctx, OPT_HEADS_FUSED) == (1 if fused else 0)
    batch = h.shape[0]
    dev = torch.device("cuda")
    th = torch.from_numpy(h).to(dev).to(torch.bfloat16)
    ids = torch.full((batch, n, k), -5, dtype=torch.int32, device=dev)
    lp = torch.zeros((batch, n, k), dtype=torch.float32, device=dev)
    V = dec.model.codec_vocab
    lg = torch.zeros((batch, n, V), dtype=torch.float32, device=dev) if want_logits else None
    lse = torch.zeros((batch, n), dtype=torch.float32, device=dev) if want_lse else None
    mtp.mtp_heads_topk(dec.ctx, batch, th, 1, n, k, ids, lp, lg, lse)
    torch.cuda.synchronize()
    return (ids.cpu().numpy(), lp.cpu().numpy(), None if lg is None else lg.cpu().numpy(),
            None if lse is None else lse.cpu().numpy())


def _check(h, w, model, n, k, ids, lp, lg, lse, rows):
    wd = {name: np.asarray(t, np.float64) for name, t in w.items()}
    for b in rows:
        ref = S.head_logits(h[b].astype(np.float64), wd, n, model.ln_eps)
        assert_logits_close(lg[b], ref, f"row {b}")
        _, ref_lse = S.log_softmax(ref)
        assert np.abs(lse[b] - ref_lse).max() < 2e-2
        r_ids, r_vals = S.top_k_rows(logp32(lg[b], lse[b]), k)
        assert np.array_equal(ids[b], r_ids), f"row {b}: top-k ids"
        assert np.array_equal(lp[b].view(np.uint32), r_vals.view(np.uint32)), f"row {b}: top-k scores"
        ref_lp32 = (ref - ref_lse[:, None]).astype(np.float32)
        o_ids, _ = S.top_k_rows(ref_lp32, k)
        gaps = S.topk_gap(ref_lp32, k)
        for i in range(n):
            if gaps[i] > MARGIN:
                assert set(o_ids[i].tolist()) == set(ids[b, i].tolist())


@pytest.mark.parametrize("batch,n,k", [(9, 1, 1), (130, 4, 4), (256, 8, 16), (40, 3, 25), (300, 2, 32),
                                       (128, 5, 7)])
def test_fused_heads_parity(batch, n, k):
    """Tiles of 128 rows with ragged tails, every candidate bucket (4, 8, 16, 32), several chunks."""
    model = synth.VALLE
    dec, w = decoder(model, max_batch=1, max_ctx=128)
    try:
        h = synth.make_hidden(batch, model.d_model, seed=100 + batch)
        ids, lp, lg, lse = _heads(dec, h, n, k)
        rows = sorted(set(list(range(0, batch, 13)) + [batch - 1, min(batch - 1, 127), min(batch - 1, 128)]))
        _check(h, w, model, n, k, ids, lp, lg, lse, rows)
    finally:
        dec.close()


def test_fused_equals_unfused_path():
    """Same rows through both paths: logits within 1e-4 (summation order differs), and each path's
    top-k exact on its own scores (checked in _check); ids equal wherever the fused scores have a clear gap."""
    model = synth.VALLE
    dec, w = decoder(model, max_batch=1, max_ctx=128)
    try:
        h = synth.make_hidden(96, model.d_model, seed=7)
        f = _heads(dec, h, 4, 8, fused=True)
        u = _heads(dec, h, 4, 8, fused=False)
        assert np.abs(f[2] - u[2]).max() < 1e-4
        assert np.abs(f[3] - u[3]).max() < 1e-4
        for b in range(96):
            sc = logp32(f[2][b], f[3][b])
            gaps = S.topk_gap(sc, 8)
            for i in range(4):
                if gaps[i] > 1e-3:
                    assert set(f[0][b, i].tolist()) == set(u[0][b, i].tolist())
    finally:
        dec.close()


def test_outputs_optional():
    """Without the logits and lse outputs the candidates are the same bits."""
    model = synth.VALLE
    dec, w = decoder(model, max_batch=1, max_ctx=128)
    try:
        h = synth.make_hidden(140, model.d_model, seed=11)
        full = _heads(dec, h, 8, 16)
        bare = _heads(dec, h, 8, 16, want_logits=False, want_lse=False)
        assert np.array_equal(full[0], bare[0])
        assert np.array_equal(full[1].view(np.uint32), bare[1].view(np.uint32))
    finally:
        dec.close()


def test_tiny_model_and_ties():
    """d = 256 (four k-chunks, fewer than the ring's stages); head weights zero and biases from a
    few levels, so every logit of a row equals a bias and whole slices tie: the candidates must be
    the lowest ids of the highest level, in id order, with logp = bias - lse."""
    model = synth.TINY_BF16
    w = dict(synth.make_weights(model))
    V = model.codec_vocab
    w["w_heads"] = np.zeros_like(w["w_heads"])
    levels = np.array([0.0, 0.5, 1.0], np.float32)
    idx = (np.arange(model.n_heads_max * V) * 7919) % 3
    idx[::97] = 2
    w["b_heads"] = levels[idx].astype(np.float32).reshape(model.n_heads_max, V)
    mtp = lib_module()
    dec = mtp.MTPDecoder(model, w, synth.weight_names(model), synth.is_matrix, 1, 128)
    try:
        h = synth.make_hidden(20, model.d_model, seed=3)
        for k in (4, 16, 32):
            ids, lp, lg, lse = _heads(dec, h, 8, k)
            for b in range(20):
                sc = logp32(lg[b], lse[b])
                r_ids, r_vals = S.top_k_rows(sc, k)
                assert np.array_equal(ids[b], r_ids)
                assert np.array_equal(lp[b].view(np.uint32), r_vals.view(np.uint32))
                bias = w["b_heads"].reshape(model.n_heads_max, V)
                for i in range(8):
                    top = np.nonzero(bias[i] == 1.0)[0][:k]
                    assert ids[b, i, :len(top)].tolist() == top.tolist()
    finally:
        dec.close()


def test_decode_steps_with_fused_heads():
    """Batched decode steps (B = 12, n = 4, top-4) with the fused heads (option 2) against the same
    teacher-forced steps with the GEMM + selection top-k (option 0) and the oracle: logits within 5e-4
    of each other (two summation orders of the same bf16 hi/lo products over d = 1024; logits up to ~4)
    and within the bf16 bar of the oracle; each run's candidates exact on its own logp
    rows; paths equal wherever the candidates are."""
    from oracle.mtp import MTPOracle
    mtp = lib_module()
    model = synth.VALLE
    B, n, k, steps = 12, 4, 4, 4
    prompts = [synth.make_prompt(300 + b, 20 + 3 * b, 60 + 5 * b, model.phone_vocab) for b in range(B)]
    runs = []
    w = None
    for opt in (2, 0):
        dec, w = decoder(model, max_batch=B, max_ctx=256)
        try:
            mtp.mtp_set_option(dec.ctx, OPT_HEADS_FUSED, opt)
            assert mtp.mtp_get_option(dec.ctx, OPT_HEADS_FUSED) == opt
            for b, (ph, ac) in enumerate(prompts):
                dec.prefill(b, ph, ac, 64)
            rec = []
            for t in range(steps):
                if t:  # teacher-forced: both runs feed the same tokens (the first run's path)
                    for b in range(B):
                        mtp.mtp_set_teacher_tokens(dec.ctx, b, runs[0][t - 1][3][b] if opt == 0 else rec[-1][3][b])
                dec.decode_step(n, k)
                lg, lse = dec.logits(n)
                ids, lp, path = dec.lattice(n, k)
                rec.append((lg.copy(), lse.copy(), (ids.copy(), lp.copy()), path.copy()))
            runs.append(rec)
        finally:
            dec.close()
    o = MTPOracle(model, w)
    ph, ac = prompts[0]
    o.prefill(ph, ac, 64)
    assert_logits_close(runs[0][0][0][0], o.step(n, k).logits, "slot 0, step 0")
    for t in range(steps):
        (lg_f, lse_f, (ids_f, lp_f), path_f), (lg_u, lse_u, (ids_u, lp_u), path_u) = runs[0][t], runs[1][t]
        assert np.abs(lg_f - lg_u).max() < 5e-4
        for b in range(B):
            r_ids, r_vals = S.top_k_rows(logp32(lg_f[b], lse_f[b]), k)
            assert np.array_equal(ids_f[b], r_ids), f"step {t} slot {b}"
            assert np.array_equal(lp_f[b].view(np.uint32), r_vals.view(np.uint32))
            if np.array_equal(ids_f[b], ids_u[b]):
                assert np.array_equal(path_f[b], path_u[b])

"""The allocation-free attention entry point against the oracle and the workspace one.

mtp_attention_noalloc serves callers that must not allocate GPU memory while
they run (for example a real-time audio callback, where cudaMalloc can block
or synchronise the device); its scratch is a fixed array inside the library.
Its output is checked against the oracle's causal attention (the attention
tests' 1e-4 bar) and must be bit-identical to mtp_attention's: both run the
same kernel with the same split count and merge order.
This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes alone in a fresh process."""
import numpy as np
import pytest

import synth
from oracle.model import causal_attention

pytestmark = pytest.mark.gpu

H, HD, LAYERS, PAGE = 4, 64, 2, 64
ATOL = 1e-4  # the attention tests' bar


def _inputs(groups, rpg, ctx, seed):
    import torch
    pages_per_seq = max(ctx) // PAGE + 2
    n_pages = groups * pages_per_seq + 1
    pool = synth.round_bf16(synth.normal(seed, "na_pool", n_pages * LAYERS * 2 * H * PAGE * HD)
                            .astype(np.float32))
    perm = np.argsort(synth.uniform(seed, "na_perm", n_pages))
    table = perm[:groups * pages_per_seq].reshape(groups, pages_per_seq).astype(np.int32)
    rows = groups * rpg
    q = synth.normal(seed, "na_q", rows * H * HD).astype(np.float32).reshape(rows, H * HD)
    row_seq = np.repeat(np.arange(groups, dtype=np.int32), rpg)
    row_pos = np.concatenate([np.arange(c - rpg, c) for c in ctx]).astype(np.int32)
    dev = torch.device("cuda")
    bits = (pool.view(np.uint32) >> 16).astype(np.uint16).view(np.int16)
    t = {name: torch.from_numpy(arr).to(dev) for name, arr in
         (("pool", bits), ("q", q), ("table", table), ("seq", row_seq), ("pos", row_pos))}
    # the oracle's attention of every row over its slot's keys/values of layer 1
    pool5 = pool.reshape(n_pages, LAYERS, 2, H, PAGE, HD)
    ref = np.zeros((rows, H, HD))
    for g in range(groups):
        logical = np.concatenate([pool5[table[g, p], 1] for p in range(pages_per_seq)], axis=2)
        k = logical[0].transpose(1, 0, 2).astype(np.float64)
        v = logical[1].transpose(1, 0, 2).astype(np.float64)
        rs = slice(g * rpg, (g + 1) * rpg)
        ref[rs] = causal_attention(q[rs].reshape(rpg, H, HD).astype(np.float64), k, v, row_pos[rs],
                                   np.arange(k.shape[0]))
    return t, rows, pages_per_seq, ref.reshape(rows, H * HD)


def _args(mtp, t, rows, rpg, pages_per_seq, max_keys, out):
    return mtp.attention_args(rows=rows, rows_per_group=rpg, n_heads=H, page_size=PAGE, layers=LAYERS, layer=1,
                              bt_stride=pages_per_seq, max_keys=max_keys, q=t["q"], kv_pool=t["pool"],
                              block_table=t["table"], row_seq=t["seq"], row_pos=t["pos"], out=out)


def test_noalloc_matches_workspace_entry_point():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2410_13839_gb300 import build
    build.build()
    from paper_2410_13839_gb300 import mtp

    stream = torch.cuda.current_stream()
    for case, (groups, rpg, ctx) in enumerate([(1, 4, [1039]), (3, 2, [300, 77, 513])]):
        t, rows, pps, oracle_out = _inputs(groups, rpg, ctx, seed=50 + case)
        ref = torch.zeros((rows, H * HD), dtype=torch.float32, device="cuda")
        args = _args(mtp, t, rows, rpg, pps, max(ctx), ref)
        nbytes = mtp.mtp_attention_workspace_bytes(args)
        ws = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
        mtp.mtp_attention(args, ws, nbytes, stream)
        for call in range(2):  # two calls in a row share the fixed scratch
            out = torch.full((rows, H * HD), -3.0, dtype=torch.float32, device="cuda")
            mtp.mtp_attention_noalloc(_args(mtp, t, rows, rpg, pps, max(ctx), out), stream)
            torch.cuda.synchronize()
            err = np.abs(out.cpu().numpy().astype(np.float64) - oracle_out).max()
            assert err <= ATOL, f"case {case} call {call}: {err} from the oracle"
            assert torch.equal(out, ref), f"case {case} call {call}: differs from mtp_attention"


def test_noalloc_rejects_calls_beyond_the_fixed_scratch():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2410_13839_gb300 import mtp
    t, rows, pps, _ = _inputs(1, 1, [70], seed=7)
    out = torch.zeros((rows, H * HD), dtype=torch.float32, device="cuda")
    big = _args(mtp, t, rows, 1, pps, 70, out)
    big.rows = 8192          # 8192 single-row groups: far more split partials than the array holds
    big.n_heads = 64
    assert mtp.mtp_attention_workspace_bytes(big) > 4 << 20
    with pytest.raises(mtp.MTPError) as e:
        mtp.mtp_attention_noalloc(big, torch.cuda.current_stream())
    assert e.value.code == -1 and "scratch" in str(e.value)

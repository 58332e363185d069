"""GPU parity of the tensor-core (tcgen05) prefill attention over the paged,
swizzled bf16 cache (Sec. III-A: every prompt position attends to itself and
the positions before it) against the oracle's causal attention.

Rows form tiles of 128; a tile may hold rows of several slots (a prefill pass
packs many prompts), inactive rows and a ragged tail.  Keys are cut into items
of 128 and spread over splits whose partials are merged; the cases put slot
ends just below, on and past item and page edges, use every page size, long
contexts and more splits than items."""
import numpy as np
import pytest

import synth
from oracle.model import causal_attention

from gpu_util import lib_module

pytestmark = pytest.mark.gpu

H, HD, LAYERS = 4, 64, 2


def swizzle_rows(pool):
    """The cache layout: 16-byte chunk c (8 bf16) of row t of a page stored at chunk c ^ (t mod 8)."""
    out = np.empty_like(pool)
    P = pool.shape[-2]
    for t in range(P):
        for c in range(8):
            cs = c ^ (t & 7)
            out[..., t, 8 * cs:8 * cs + 8] = pool[..., t, 8 * c:8 * c + 8]
    return out


def _run(rows_spec, page_size, ctx_of, max_keys=None, seed=0, layer=1, calls=2):
    """rows_spec: list of (slot, position) per row, slot -1 = inactive; ctx_of[slot] = cached keys."""
    import torch
    mtp = lib_module()
    slots = len(ctx_of)
    max_ctx = max(ctx_of)
    pages_per_seq = (max_ctx + page_size - 1) // page_size + 1
    n_pages = slots * pages_per_seq + 3
    pool = synth.round_bf16(synth.normal(seed, "pool", n_pages * LAYERS * 2 * H * page_size * HD)
                            .astype(np.float32)).reshape(n_pages, LAYERS, 2, H, page_size, HD)
    perm = np.argsort(synth.uniform(seed, "perm", n_pages))        # scattered physical pages
    table = np.full((slots, pages_per_seq), -1, np.int32)
    for s in range(slots):
        used = (ctx_of[s] + page_size - 1) // page_size
        table[s, :used] = perm[s * pages_per_seq:s * pages_per_seq + used]
    rows = len(rows_spec)
    q = synth.normal(seed, "q", rows * H * HD).astype(np.float32).reshape(rows, H, HD)
    row_seq = np.array([s for s, _ in rows_spec], np.int32)
    row_pos = np.array([p for _, p in rows_spec], np.int32)
    dev = torch.device("cuda")
    bits = (swizzle_rows(pool).view(np.uint32) >> 16).astype(np.uint16)
    t_pool = torch.from_numpy(bits.view(np.int16)).to(dev)
    t_q = torch.from_numpy(q.reshape(rows, H * HD)).to(dev)
    t_tab = torch.from_numpy(table).to(dev)
    t_seq = torch.from_numpy(row_seq).to(dev)
    t_pos = torch.from_numpy(row_pos).to(dev)
    out = torch.full((rows, H * HD), -7.0, dtype=torch.float32, device=dev)
    args = mtp.attention_args(rows=rows, rows_per_group=1, n_heads=H, page_size=page_size, layers=LAYERS,
                              layer=layer, bt_stride=pages_per_seq, max_keys=max_keys or max_ctx,
                              q=t_q, kv_pool=t_pool, block_table=t_tab, row_seq=t_seq, row_pos=t_pos, out=out)
    nbytes = mtp.mtp_attention_tc_workspace_bytes(args)
    assert nbytes > 0
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    refs = {}
    for s in set(int(x) for x in row_seq if x >= 0):
        used = (ctx_of[s] + page_size - 1) // page_size
        logical = np.concatenate([pool[table[s, p], layer] for p in range(used)], axis=2)
        k = logical[0].transpose(1, 0, 2).astype(np.float64)[:ctx_of[s]]   # [T, H, HD]
        v = logical[1].transpose(1, 0, 2).astype(np.float64)[:ctx_of[s]]
        idx = np.nonzero(row_seq == s)[0]
        refs[s] = (idx, causal_attention(q[idx].astype(np.float64), k, v, row_pos[idx], np.arange(k.shape[0])))
    for _ in range(calls):        # the merge counters come back to zero: a second call agrees
        out.fill_(-7.0)
        mtp.mtp_attention_tc(args, ws, nbytes, torch.cuda.current_stream())
        torch.cuda.synchronize()
        got = out.cpu().numpy().reshape(rows, H, HD)
        assert np.all(got[row_seq < 0] == -7.0), "inactive row was written"
        for s, (idx, ref) in refs.items():
            err = np.abs(got[idx] - ref).max()
            assert err < 1e-4, f"slot {s}: max error {err}"
    return got


def _chunk(slot, p0, m):
    return [(slot, p0 + i) for i in range(m)]


@pytest.mark.parametrize("page", [16, 32, 64, 128])
def test_first_chunk_causal_within_the_tile(page):
    """One slot, positions 0..127: every key is a row of the tile itself."""
    _run(_chunk(0, 0, 128), page, [128])


def test_valle_second_chunk():
    """Positions 161..288 of a 289-position prompt (64 + 225), pages of 64: three items, the last partial."""
    _run(_chunk(0, 161, 128), 64, [289])


@pytest.mark.parametrize("ctx", [127, 128, 129, 255, 256, 257])
def test_item_edges(ctx):
    """Slot ends just below, on and past 128-key item edges; rows are the last positions."""
    m = min(ctx, 40)
    _run(_chunk(0, ctx - m, m), 32, [ctx])


def test_one_key():
    _run([(0, 0)], 64, [1])


def test_several_slots_per_tile_ragged():
    """300 rows (three tiles, the last ragged): slots interleaved in runs of 8 positions, as a
    prefill pass packs prompts; pages of 16."""
    ctx = [150, 310, 97]
    spec, nxt = [], [0, 0, 0]
    order = [0, 1, 2, 1, 1, 0, 2, 1] * 8   # 64 runs of 8 rows at most: a bounded loop
    for s in order:
        if nxt[s] + 8 <= ctx[s] and len(spec) + 8 <= 296:
            spec += _chunk(s, nxt[s], 8)
            nxt[s] += 8
    spec += [(-1, 0)] * (300 - len(spec))
    _run(spec, 16, ctx)


def test_many_slots_long_contexts_and_inactive_rows():
    """16 slots of 8 rows in one tile, contexts up to 2000 (pages of 128), some rows inactive."""
    ctx = [50 + 131 * s for s in range(15)] + [2000]
    spec = []
    for s in range(16):
        spec += _chunk(s, ctx[s] - 8, 8)
    for r in (3, 64, 65, 127):
        spec[r] = (-1, 0)
    _run(spec, 128, ctx, seed=3)


def test_spare_splits():
    """max_keys far above the contexts: splits without items still merge correctly."""
    _run(_chunk(0, 100, 28) + _chunk(1, 0, 20), 64, [128, 20], max_keys=6000, seed=5)


def test_rejects_bad_arguments():
    import torch
    mtp = lib_module()
    t = torch.zeros(64, dtype=torch.float32, device="cuda")
    i = torch.zeros(4, dtype=torch.int32, device="cuda")
    args = mtp.attention_args(rows=1, rows_per_group=1, n_heads=1, page_size=48, layers=1, layer=0, bt_stride=1,
                              max_keys=1, q=t, kv_pool=t, block_table=i, row_seq=i, row_pos=i, out=t)
    assert mtp.mtp_attention_tc_workspace_bytes(args) == 0
    ws = torch.zeros(1 << 16, dtype=torch.uint8, device="cuda")
    with pytest.raises(mtp.MTPError):
        mtp.mtp_attention_tc(args, ws, 1 << 16, torch.cuda.current_stream())


OPT_PREFILL_TC = 10


@pytest.mark.parametrize("model_name,page_size", [("VALLE", 64), ("TINY_BF16", 16)])
def test_prefill_passes_tc_equal_split_key_kernel(model_name, page_size):
    """Prefill (several 128-row chunks) and prefill_pending (prompts of several slots packed in
    one pass) with the tensor-core attention against the split-key kernel and the oracle: the
    first step's logits within 1e-3 of each other and within the bf16 bar of the oracle."""
    from oracle.mtp import MTPOracle
    from gpu_util import assert_logits_close, decoder
    mtp = lib_module()
    model = getattr(synth, model_name)
    prompts = [synth.make_prompt(20 + b, 30 + 11 * b, 200 + 37 * b, model.phone_vocab) for b in range(3)]
    outs = []
    for tc in (1, 0):
        dec, w = decoder(model, max_batch=3, max_ctx=700, page_size=page_size)
        try:
            mtp.mtp_set_option(dec.ctx, OPT_PREFILL_TC, tc)
            assert mtp.mtp_get_option(dec.ctx, OPT_PREFILL_TC) == tc
            dec.prefill(0, *prompts[0], 40)       # chunks of 128 positions of one slot
            for b in (1, 2):                      # packed passes of both slots' prompts
                dec.admit(b, *prompts[b], 40)
            assert mtp.mtp_prefill_pending(dec.ctx) >= 1
            dec.decode_step(4, 4)
            outs.append(dec.logits(4)[0].copy())
        finally:
            dec.close()
        if tc:
            o = MTPOracle(model, w)
            for b, (ph, ac) in enumerate(prompts):
                o.prefill(ph, ac, 40)
                assert_logits_close(outs[0][b], o.step(4, 4).logits, f"slot {b}")
    assert np.abs(outs[0] - outs[1]).max() <= 1e-3

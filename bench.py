"""Benchmark of the MTP decode path on one VALL-E-sized workload.

Workload (one "step"): batch 1, prompt = 64 phonemes + 225 acoustic codes,
prefill, then decode 750 codec tokens with n = 4 heads and top_k = 4
(ceil(750 / 4) = 188 decode steps) -- whole-job codec tokens/s.  Synthetic
seeded weights and prompts (synth); the 302 MB of weights per decode step
are larger than L2, so no flush is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line.  --impl reference times the CPU oracle on the host
cores (a bounded sample of the same workload).  Under torchrun (N > 1) every
rank runs an independent replica (no collective on the data path); the
value is all ranks' tokens over the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import platform
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

N_PH, N_AC, GEN, N_HEADS, TOP_K, BATCH = 64, 225, 750, 4, 4, 1
WORKLOAD = "VALL-E-sized AR decode: 12 layers, d=1024, 16 heads, FFN 4096, bf16; B=1, prompt 64+225, 750 tokens, n=4, top_k=4"
METRIC = "codec tokens/s at B=1 (n=4 heads, top_k=4)"
MODEL = synth.VALLE
MAX_CTX = N_PH + N_AC + GEN + MODEL.n_heads_max + 8


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        p = json.load(open(path))
        return float(p["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def _config():
    return {"workload": WORKLOAD, "batch": BATCH, "prompt": [N_PH, N_AC], "generate": GEN,
            "n_heads": N_HEADS, "top_k": TOP_K, "page_size": 64,
            "l2": "inputs larger than L2: 302 MB of weights streamed per decode step (L2 129 MB)",
            "parallelism": "replicas"}


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(x: float, dist=None, device="cuda") -> float:
    """The largest x over all ranks (the slowest rank's time); x itself on one rank."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(world: int, steps: int, seconds: float) -> float:
    """Whole-job throughput: every rank's generated tokens over the slowest rank's time."""
    return world * steps * GEN * BATCH / seconds


def _kernel_bytes(d, F, V, L, n, wb, ctx_keys, fed):
    """Algorithmic bytes per launch of each kernel class (weights + parameters; keys/values)."""
    return {
        "attn_block": (4 * d * d) * wb + (3 * d + d + 2 * d) * 4 + ctx_keys * d * 2 * 2 + fed * d * 2 * 2,
        "mlp": 2 * F * d * wb + (F + d + 2 * d) * 4,
        "heads": n * V * d * wb + n * V * 4 + 2 * d * 4,
        # the persistent kernel: the fed rows' embedding and all L blocks of one pass
        "step": L * ((4 * d * d + 2 * F * d) * wb + (3 * d + d + F + d + 4 * d) * 4
                     + ctx_keys * d * 2 * 2 + fed * d * 2 * 2) + fed * d * (wb + 4),
    }


def _decode_bytes_total(d, F, V, L, n, wb, prompt_len, gen):
    """Algorithmic bytes of all decode steps of one generation (weights, heads, KV read + write)."""
    weights = L * ((3 * d * d + d * d + 2 * d * F) * wb + (3 * d + d + F + d + 4 * d) * 4)
    heads = n * V * d * wb + n * V * 4 + 2 * d * 4
    total, cached, produced = 0, prompt_len, 0
    fed = 0
    while produced < gen:
        step = heads
        if fed:
            step += weights + L * (cached + fed) * d * 4 + L * fed * d * 4
            cached += fed
        a = min(n, gen - produced)
        produced += a
        fed = a
        total += step
    return total


B32 = 32
B32_WORKLOAD = ("VALL-E-sized batched serving: B=32, prompts U[32,128] phonemes + U[150,450] acoustic, "
                "generation U[375,1500] with per-sequence EOS, n=4, top_k=4")


def b32_sequences(batch=B32):
    """Prompt lengths, prompts and generation budgets of the batched-serving workload."""
    seqs = []
    for i in range(batch):
        n_ph = synth.make_lengths(i, 32, 128, "serve_phonemes")
        n_ac = synth.make_lengths(i, 150, 450, "serve_acoustic")
        gen = synth.make_lengths(i, 375, 1500, "serve_generate")
        ph, ac = synth.make_prompt(i, n_ph, n_ac, MODEL.phone_vocab)
        seqs.append((ph, ac, gen))
    return seqs


def _batched_decode_bytes(prompt_lens, gens, d, F, V, L, n, wb):
    """Algorithmic bytes of the decode steps of a batch run in lockstep: weights and
    heads once per step, cached keys/values read and the fed rows' written per active sequence."""
    weights = L * ((3 * d * d + d * d + 2 * d * F) * wb + (3 * d + d + F + d + 4 * d) * 4)
    heads = n * V * d * wb + n * V * 4 + 2 * d * 4
    cached, produced, fed = list(prompt_lens), [0] * len(gens), [0] * len(gens)
    total = 0
    while any(p < g for p, g in zip(produced, gens)):
        kv, any_fed = 0, False
        for i, g in enumerate(gens):
            if produced[i] >= g:
                continue
            if fed[i]:
                kv += L * (cached[i] + fed[i]) * d * 4 + L * fed[i] * d * 4
                cached[i] += fed[i]
                any_fed = True
            a = min(n, g - produced[i])
            produced[i] += a
            fed[i] = a
        total += heads + (weights + kv if any_fed else 0)
    return total


def run_b32(mtp, stream, warmup, steps, batch=B32, interleaved=False):
    """Whole-job codec tokens/s of the batched-serving workload on this GPU (prefill + decode).

    The prompts are admitted (mtp_admit) and run together by mtp_prefill_pending (many slots'
    prompt rows per pass), then mtp_generate decodes.  With `interleaved` the job also runs once
    with the prompts prefilled inside the decode steps' lane instead (mtp_generate directly)."""
    import torch
    seqs = b32_sequences(batch)
    max_ctx = max(len(p) + len(a) + g for p, a, g in seqs) + MODEL.n_heads_max + 8
    w = synth.make_weights(MODEL)
    dec = mtp.MTPDecoder(MODEL, w, synth.weight_names(MODEL), synth.is_matrix, batch, max_ctx, stream=stream)
    ctx = dec.ctx
    dev = [(torch.from_numpy(p).cuda(), torch.from_numpy(a).cuda(), g) for p, a, g in seqs]
    lens = torch.zeros(batch, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()

    def job(ev=None, together=True):
        if ev:
            ev[0].record(stream)
        for b, (p, a, g) in enumerate(dev):
            mtp.mtp_admit(ctx, b, p, a, g)
        if together:
            mtp.mtp_prefill_pending(ctx)
        if ev:
            ev[1].record(stream)
        n_steps = mtp.mtp_generate(ctx, N_HEADS, TOP_K, None, 0, lens)
        if ev:
            ev[2].record(stream)
        return n_steps

    for _ in range(warmup):
        job()
    torch.cuda.synchronize()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    dsteps = 0
    for i in range(steps):
        dsteps += job(evs[i])
    torch.cuda.synchronize()
    tokens = int(lens.sum().item())
    total_ms = sum(e[0].elapsed_time(e[2]) for e in evs)
    decode_ms = sum(e[1].elapsed_time(e[2]) for e in evs) / steps
    prefill_ms = sum(e[0].elapsed_time(e[1]) for e in evs) / steps
    d, F, V, L = MODEL.d_model, MODEL.d_ffn, MODEL.codec_vocab, MODEL.layers
    dec_bytes = _batched_decode_bytes([len(p) + len(a) for p, a, _ in seqs], [g for _, _, g in seqs],
                                      d, F, V, L, N_HEADS, 2)
    peak, peak_kind = _peaks()
    batched = mtp.mtp_get_option(ctx, mtp.MTP_OPT_BATCHED)
    inter = None
    if interleaved:  # the same job with every prompt prefilled in the lane of the decode steps
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        isteps = job(ev, together=False)
        torch.cuda.synchronize()
        inter = {"ms_per_job": ev[0].elapsed_time(ev[2]), "steps": isteps,
                 "tokens_per_s": int(lens.sum().item()) / (ev[0].elapsed_time(ev[2]) / 1e3)}
    dec.close()
    return {"value": tokens * steps / (total_ms / 1e3), "unit": "codec tokens/s", "batch": batch,
            "workload": B32_WORKLOAD.replace("B=32", "B=%d" % batch), "tokens_per_job": tokens, "jobs": steps, "warmup_jobs": warmup,
            "ms_per_job": total_ms / steps, "prefill_ms": prefill_ms, "decode_ms": decode_ms,
            "decode_steps_per_job": dsteps // steps, "decode_tokens_per_s": tokens / (decode_ms / 1e3),
            "path": "batched (tensor-core projections)" if batched else "fused 8-row passes",
            "prefill": "prompts admitted, then run together (mtp_prefill_pending: passes of up to all batched rows)",
            "interleaved": inter,
            "decode_roofline": {"decode_bytes": dec_bytes, "achieved_gbs": dec_bytes / (decode_ms / 1e3) / 1e9,
                                "peak": peak, "peak_source": peak_kind,
                                "frac": dec_bytes / (decode_ms / 1e3) / 1e9 / peak}}


SWEEP_GEN = 1500


C5_BATCH, C5_N, C5_K, C5_LATTICES = 256, 8, 16, 10000


def c5_lattices(count: int, n: int, k: int, vocab: int, seed: int = 5):
    """Seeded lattices of the microbenchmark shape: per (lattice, position) k distinct ids
    (an arithmetic progression mod vocab with a step coprime to it) and log-uniform scores
    sorted in descending order, as a top-k would give them."""
    rng = np.random.default_rng(seed)
    start = rng.integers(0, vocab, size=(count, n, 1))
    step = rng.integers(1, vocab, size=(count, n, 1))
    bad = np.gcd(step, vocab) != 1
    while bad.any():
        step[bad] = rng.integers(1, vocab, size=int(bad.sum()))
        bad = np.gcd(step, vocab) != 1
    ids = ((start + step * np.arange(k)) % vocab).astype(np.int32)
    lp = -np.sort(-np.log1p(-rng.random((count, n, k))), axis=2).astype(np.float32)
    return ids, lp


def run_c5(mtp, stream):
    """The isolated head + Viterbi microbenchmark: n=8 heads with log-softmax and top-16
    on 256 bf16 hidden rows N(0,1) (VALL-E-sized heads, in a context whose row buffers
    hold all 256 rows: one heads launch per call), and Viterbi with acceptance over 10^4
    lattices of 8 positions x 16 candidates.  CUDA events, 3 warm-up calls; head bytes =
    the 8 heads' weights once per call.  The heads call asks for the candidates and lse
    only (the logits stay on chip)."""
    import torch
    d, V = MODEL.d_model, MODEL.codec_vocab
    w = synth.make_weights(MODEL)
    dec = mtp.MTPDecoder(MODEL, w, synth.weight_names(MODEL), synth.is_matrix, C5_BATCH // MODEL.n_heads_max, 64,
                         stream=stream)
    ctx = dec.ctx
    h = torch.from_numpy(synth.make_hidden(C5_BATCH, d, seed=C5_BATCH)).cuda().to(torch.bfloat16)
    ids = torch.zeros((C5_BATCH, C5_N, C5_K), dtype=torch.int32, device="cuda")
    lp = torch.zeros((C5_BATCH, C5_N, C5_K), dtype=torch.float32, device="cuda")
    lse = torch.zeros((C5_BATCH, C5_N), dtype=torch.float32, device="cuda")
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    calls = 20
    for _ in range(3):
        mtp.mtp_heads_topk(ctx, C5_BATCH, h, 1, C5_N, C5_K, ids, lp, None, lse)
    torch.cuda.synchronize()
    ev[0].record(stream)
    for _ in range(calls):
        mtp.mtp_heads_topk(ctx, C5_BATCH, h, 1, C5_N, C5_K, ids, lp, None, lse)
    ev[1].record(stream)
    torch.cuda.synchronize()
    heads_s = ev[0].elapsed_time(ev[1]) / 1e3 / calls
    c_ids, c_lp = c5_lattices(C5_LATTICES, C5_N, C5_K, V)
    t_ids, t_lp = torch.from_numpy(c_ids).cuda(), torch.from_numpy(c_lp).cuda()
    t_q = torch.from_numpy(synth.transition_log_q(V)).cuda()
    path = torch.zeros((C5_LATTICES, C5_N), dtype=torch.int32, device="cuda")
    acc = torch.zeros(C5_LATTICES, dtype=torch.int32, device="cuda")
    vs = torch.cuda.current_stream()
    for _ in range(3):
        mtp.mtp_viterbi(C5_LATTICES, C5_N, C5_K, V, MODEL.eos_id, t_ids, t_lp, t_q, None, path, None, acc, None, vs)
    torch.cuda.synchronize()
    ev[2].record(vs)
    for _ in range(calls):
        mtp.mtp_viterbi(C5_LATTICES, C5_N, C5_K, V, MODEL.eos_id, t_ids, t_lp, t_q, None, path, None, acc, None, vs)
    ev[3].record(vs)
    torch.cuda.synchronize()
    vit_s = ev[2].elapsed_time(ev[3]) / 1e3 / calls
    dec.close()
    head_bytes = C5_N * V * d * 2
    # algorithmic bytes of one heads call: the head weights and biases, the hidden rows (bf16),
    # the candidates (ids + logp) and lse written
    call_bytes = head_bytes + C5_N * V * 4 + C5_BATCH * d * 2 + C5_BATCH * C5_N * (C5_K * 8 + 4)
    flops = 2.0 * C5_BATCH * C5_N * V * d
    gathers = C5_LATTICES * (C5_N - 1) * C5_K * C5_K
    peak, peak_src = _peaks()
    return {"workload": "isolated heads + Viterbi: 256 bf16 hidden rows N(0,1), n=8 heads x V=1025 with "
                        "log-softmax and top-16; Viterbi + acceptance over 10^4 lattices of 8 x 16",
            "heads_topk_us": heads_s * 1e6, "heads_gbs": head_bytes / heads_s / 1e9,
            "heads_tflops": flops / heads_s / 1e12,
            "heads_roofline": {"bound": "hbm", "achieved": call_bytes / heads_s / 1e9, "peak": peak,
                               "unit": "GB/s", "frac": call_bytes / heads_s / 1e9 / peak,
                               "peak_source": peak_src, "algorithmic_bytes_per_call": call_bytes,
                               "note": "one call = row conversion, LN_f pack and the fused heads kernel"},
            "viterbi_us": vit_s * 1e6,
            "viterbi_lattices_per_s": C5_LATTICES / vit_s,
            "viterbi_roofline": {
                "bound": "l2_tag_requests", "achieved": gathers / vit_s / 1e9, "peak": L2_TAG_REQUESTS_PEAK,
                "unit": "G gathers/s", "frac": gathers / vit_s / 1e9 / L2_TAG_REQUESTS_PEAK,
                "traffic": VITERBI_C5_TAG_REQUESTS, "gathers_per_call": gathers,
                "peak_source": "ncu: lts__t_tag_requests.sum.per_second / its % of peak (GB300)"}}


# The stand-alone Viterbi gathers (n-1) k^2 transition scores per lattice, 4 bytes
# each at arbitrary ids from a table resident in L2: one L2 tag lookup per
# gather, so the L2's tag-request rate bounds it.  ncu on GB300: 236 requests/ns
# at 62.5 % of peak -> 378 G requests/s; 15.1 M requests per C5 call.
L2_TAG_REQUESTS_PEAK = 378.0
VITERBI_C5_TAG_REQUESTS = 15_144_000


def run_sweep(mtp, stream):
    """Head/beam sweep on the VALL-E-sized model (B=1, prompt 64+225, 1500 tokens): tokens/s
    (prefill + decode) and mean accepted tokens per step for each (n, top_k); and the mean
    accepted tokens per step of VERIFY_GREEDY at n=4, top_k=4 (random-init heads)."""
    import torch
    w = synth.make_weights(MODEL)
    ph, ac = synth.make_prompt(0, N_PH, N_AC, MODEL.phone_vocab)
    max_ctx = N_PH + N_AC + SWEEP_GEN + MODEL.n_heads_max + 8
    rows = []
    for policy in (0, 1):
        dec = mtp.MTPDecoder(MODEL, w, synth.weight_names(MODEL), synth.is_matrix, 1, max_ctx, stream=stream,
                             accept_policy=policy)
        ctx = dec.ctx
        ph_d, ac_d = torch.from_numpy(ph).cuda(), torch.from_numpy(ac).cuda()
        lens = torch.zeros(1, dtype=torch.int32, device="cuda")
        grid = [(n, k) for n in (1, 2, 4, 8) for k in (1, 4, 8, 25)] if policy == 0 else [(4, 4)]
        for n, k in grid:
            for rep in range(2):  # the first run captures the step graph
                ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
                ev[0].record(stream)
                mtp.mtp_prefill(ctx, 0, ph_d, ac_d, SWEEP_GEN)
                steps = mtp.mtp_generate(ctx, n, k, None, 0, lens)
                ev[1].record(stream)
                torch.cuda.synchronize()
            toks = int(lens[0].item())
            rows.append({"policy": "VERIFY_GREEDY" if policy else "ACCEPT_ALL", "n": n, "top_k": k,
                         "tokens": toks, "steps": steps, "mean_accepted": toks / max(1, steps),
                         "tokens_per_s": toks / (ev[0].elapsed_time(ev[1]) / 1e3)})
        dec.close()
    return rows


class ClockSampler:
    """nvidia-smi clock/throttle samples while the timed region runs."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        rows = [r.split(",") for r in (self.out or "").strip().splitlines() if r.count(",") >= 8]
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        sm = [float(r[1]) for r in rows]
        smax = max(float(r[2]) for r in rows)
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].strip() == "Active"})
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": reasons, "samples": len(rows)}


def cpu_model() -> str:
    """The host CPU as /proc/cpuinfo names it (model name, or implementer/part on Arm)."""
    try:
        info = open("/proc/cpuinfo").read()
    except OSError:
        return platform.machine()
    for line in info.splitlines():
        if line.lower().startswith("model name"):
            return line.split(":", 1)[1].strip()
    fields = {}
    for line in info.splitlines():
        if ":" in line:
            k, v = line.split(":", 1)
            fields.setdefault(k.strip(), v.strip())
    parts = [f"{k} {fields[k]}" for k in ("CPU implementer", "CPU part", "CPU variant") if k in fields]
    return f"{platform.machine()} ({', '.join(parts)})" if parts else platform.machine()


def _oracle_rate(max_steps: int):
    """The oracle as it stands: prefill + the first decode steps of the workload (tokens/s, sample)."""
    from oracle.mtp import MTPOracle
    w = synth.make_weights(MODEL)
    ph, ac = synth.make_prompt(0, N_PH, N_AC, MODEL.phone_vocab)
    o = MTPOracle(MODEL, w)
    t0 = time.perf_counter()
    o.prefill(ph, ac, GEN)
    recs = o.generate(N_HEADS, TOP_K, max_steps=max_steps)
    dt = time.perf_counter() - t0
    toks = sum(r.accepted for r in recs)
    return toks / dt, (f"prefill of the {N_PH + N_AC}-token prompt + first {len(recs)} decode steps "
                       f"({toks} tokens), float64 numpy, {dt:.1f} s")


def cpu_baseline(max_steps: int = 60, single_steps: int = 16):
    """The oracle on this host's cores, and on one core (a child process with one BLAS thread)."""
    value, sample = _oracle_rate(max_steps)
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    out = {"value": value, "unit": "codec tokens/s", "cores": cores, "kind": "oracle", "sample": sample,
           "cpu_model": cpu_model()}
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    try:
        res = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-rate-steps", str(single_steps)],
                             env=env, capture_output=True, text=True, timeout=600)
        one = json.loads(res.stdout.strip().splitlines()[-1])
        out["single_thread"] = {"value": one["value"], "unit": "codec tokens/s", "cores": 1, "sample": one["sample"]}
    except (subprocess.SubprocessError, ValueError, IndexError, KeyError, OSError) as e:
        out["single_thread"] = {"value": None, "error": type(e).__name__}
    return out


KERNEL_SOURCES = ("paper_2410_13839_gb300/csrc/layer_fused.cu", "paper_2410_13839_gb300/csrc/frag.cuh",
                  "paper_2410_13839_gb300/csrc/common.cuh")


def kernel_source_sha1() -> str:
    """Hash of the block kernels' sources (the ncu traffic figure is valid only for these)."""
    h = hashlib.sha1()
    for rel in KERNEL_SOURCES:
        h.update(open(os.path.join(ROOT, rel), "rb").read())
    return h.hexdigest()


def _traffic_for(kind: str):
    """DRAM bytes per launch from the committed ncu summary, if the kernel sources are unchanged.

    profiles/traffic.txt holds lines `<kernel kind> <sources sha1> <dram bytes per launch>`."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    sha = kernel_source_sha1()
    for line in open(path):
        parts = line.split()
        if len(parts) == 3 and parts[0] == kind and parts[1] == sha:
            return int(parts[2])
    return None


def run_reference(args):
    world, rank, _ = _dist()
    if rank != 0:
        return
    from oracle.mtp import MTPOracle
    w = synth.make_weights(MODEL)
    ph, ac = synth.make_prompt(0, N_PH, N_AC, MODEL.phone_vocab)
    o = MTPOracle(MODEL, w)
    o.prefill(ph, ac, GEN)
    per_step = 8    # decode steps per bench step: a bounded sample of the generation
    times, toks = [], 0
    for i in range(args.warmup + args.steps):
        if o.done:
            o.prefill(ph, ac, GEN)
        t0 = time.perf_counter()
        recs = o.generate(N_HEADS, TOP_K, max_steps=per_step)
        dt = time.perf_counter() - t0
        if i >= args.warmup:
            times.append(dt)
            toks += sum(r.accepted for r in recs)
    total = sum(times)
    value = toks / total
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "codec tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": _config(),
            "cpu_baseline": {"value": value, "unit": "codec tokens/s", "cores": cores, "kind": "oracle",
                             "sample": f"{per_step} decode steps ({per_step * N_HEADS} tokens) per bench step "
                                       "after one untimed prefill; float64 numpy oracle"},
            "e2e": {"value": value, "unit": "codec tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_ours(args):
    import torch
    world, rank, local = _dist()
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    cpu = cpu_baseline() if (rank == 0 and world == 1 and not args.no_cpu_baseline) else None

    from paper_2410_13839_gb300 import build
    build.build()
    from paper_2410_13839_gb300 import mtp

    stream = torch.cuda.Stream()
    w = synth.make_weights(MODEL)
    dec = mtp.MTPDecoder(MODEL, w, synth.weight_names(MODEL), synth.is_matrix, BATCH, MAX_CTX, stream=stream)
    ctx = dec.ctx
    ph, ac = synth.make_prompt(rank, N_PH, N_AC, MODEL.phone_vocab)
    with torch.cuda.stream(stream):
        ph_d = torch.from_numpy(ph).cuda()
        ac_d = torch.from_numpy(ac).cuda()
    stream.synchronize()
    lens = torch.zeros(BATCH, dtype=torch.int32, device="cuda")

    def one_step(ev=None):
        if ev:
            ev[0].record(stream)
        mtp.mtp_prefill(ctx, 0, ph_d, ac_d, GEN)
        if ev:
            ev[1].record(stream)
        steps = mtp.mtp_generate(ctx, N_HEADS, TOP_K, None, 0, lens)
        if ev:
            ev[2].record(stream)
        return steps

    def barrier():
        if dist:
            dist.barrier()
        torch.cuda.synchronize()

    for _ in range(args.warmup):
        one_step()
    barrier()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    with ClockSampler(local) as clk:
        start = torch.cuda.Event(enable_timing=True)
        stop = torch.cuda.Event(enable_timing=True)
        start.record(stream)
        decode_steps = 0
        for i in range(args.steps):
            decode_steps += one_step(evs[i])
        stop.record(stream)
        barrier()
    ms = start.elapsed_time(stop)
    tokens_done = int(lens.cpu()[0])
    assert tokens_done == GEN, f"generation stopped at {tokens_done} tokens"
    prefill_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    decode_ms = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
    ms = max_over_ranks(ms, dist)
    value = job_tokens_per_s(world, args.steps, ms / 1e3)

    # end to end through the public API with host buffers (pinned), copies inside the timed region
    ph_h = torch.from_numpy(ph).pin_memory()
    ac_h = torch.from_numpy(ac).pin_memory()
    out_h = torch.zeros((BATCH, GEN), dtype=torch.int32).pin_memory()
    lens_h = torch.zeros(BATCH, dtype=torch.int32).pin_memory()
    barrier()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        mtp.mtp_prefill(ctx, 0, ph_h, ac_h, GEN)
        mtp.mtp_generate(ctx, N_HEADS, TOP_K, out_h, GEN, lens_h)
    barrier()
    e2e_s = time.perf_counter() - t0
    e2e_s = max_over_ranks(e2e_s, dist)
    e2e = {"value": job_tokens_per_s(world, args.steps, e2e_s), "unit": "codec tokens/s",
           "h2d_bytes_per_step": (N_PH + N_AC) * 4, "d2h_bytes_per_step": BATCH * GEN * 4 + BATCH * 4}

    # per-kernel durations: one eager step mid-generation, events around every launch
    mtp.mtp_prefill(ctx, 0, ph_d, ac_d, GEN)
    for _ in range(GEN // N_HEADS // 2):
        mtp.mtp_decode_step(ctx, N_HEADS, TOP_K)
    state = mtp.mtp_seq_state(ctx, 0)
    prof = mtp.mtp_profile_step(ctx, N_HEADS, TOP_K)
    d, F, V, L = MODEL.d_model, MODEL.d_ffn, MODEL.codec_vocab, MODEL.layers
    kb = _kernel_bytes(d, F, V, L, N_HEADS, 2, state["len"] + state["pending"], state["pending"])
    dom = max(kb, key=lambda kind: prof[kind][0])
    per_launch_ms = prof[dom][0] / max(1, prof[dom][1])
    peak, peak_kind = _peaks()
    achieved = kb[dom] / (per_launch_ms / 1e3) / 1e9
    traffic = _traffic_for(dom)
    # the same kernel inside the graph-launched, programmatically overlapped step: %globaltimer from its
    # last CTA past the dependency wait to its last CTA's end, averaged over the step's launches
    from paper_2410_13839_gb300._lib import KERNEL_KINDS
    mtp.mtp_trace_step(ctx, N_HEADS, TOP_K)  # captures the traced step
    tr = mtp.mtp_trace_step(ctx, N_HEADS, TOP_K)
    spans = [(r[3] - r[2]) / 1e3 for r in tr if KERNEL_KINDS[int(r[0])] == dom and r[3] > r[2]]
    pipelined_us = statistics.mean(spans) if spans else None
    # the traced step by kernel kind: launches, mean time from the last CTA past the dependency wait
    # to the last CTA's end, and mean time from the previous launch's end to this one's wait
    timeline = {}
    for i, r in enumerate(tr):
        kind = KERNEL_KINDS[int(r[0])]
        t = timeline.setdefault(kind, {"launches": 0, "post_wait_us": 0.0, "gap_us": 0.0})
        t["launches"] += 1
        t["post_wait_us"] += max(0, int(r[3]) - int(r[2])) / 1e3
        if i > 0:
            t["gap_us"] += max(0, int(r[2]) - int(tr[i - 1][3])) / 1e3
    for t in timeline.values():
        t["post_wait_us"] /= t["launches"]
        t["gap_us"] /= t["launches"]
    step_span_us = (int(tr[-1][3]) - int(tr[0][1])) / 1e3 if len(tr) else None
    roofline = {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": traffic, "peak_source": peak_kind,
                "algorithmic_bytes_per_launch": kb[dom], "avg_launch_us": per_launch_ms * 1e3,
                "timing": "one eager decode step at context %d, CUDA events around each launch" % state["len"],
                "pipelined_us": pipelined_us,
                "pipelined_frac": kb[dom] / (pipelined_us / 1e6) / 1e9 / peak if pipelined_us else None}
    dec_bytes = _decode_bytes_total(d, F, V, L, N_HEADS, 2, N_PH + N_AC, GEN)
    step_roof = {"decode_bytes": dec_bytes, "decode_ms": decode_ms,
                 "achieved_gbs": dec_bytes / (decode_ms / 1e3) / 1e9,
                 "frac": dec_bytes / (decode_ms / 1e3) / 1e9 / peak,
                 "frac_of_nominal_8tbs": dec_bytes / (decode_ms / 1e3) / 1e9 / 8000.0}
    # prefill: two slot updates, then per 128-position chunk the embedding, 8 batched-path kernels per
    # layer and the last-row save; decode: the persistent step kernel (or the embedding and 2 block
    # kernels per layer), heads, selection
    per_decode_step = 3 if mtp.mtp_get_option(ctx, 9) else 3 + 2 * L
    launches_per_step = (2 + ((N_PH + N_AC + 127) // 128) * (2 + 8 * L)
                         + decode_steps // args.steps * per_decode_step)

    line = {"metric": METRIC, "value": value, "unit": "codec tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": _config(),
            "roofline": roofline, "decode_roofline": step_roof,
            "prefill_ms": prefill_ms, "decode_ms": decode_ms,
            "decode_tokens_per_s": GEN / (decode_ms / 1e3),
            "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches_per_step * args.steps,
            "clocks": clk.summary(), "kernel_ms": {k: v[0] for k, v in prof.items()},
            "step_timeline": {"span_us": step_span_us, "kinds": timeline,
                              "timing": "one graph-launched decode step, %globaltimer (mtp_trace_step)"}}
    if not args.no_c5:
        line["c5"] = run_c5(mtp, stream)
    dec.close()
    if not args.no_b32:
        line["b32"] = run_b32(mtp, stream, max(1, min(args.warmup, 2)), max(1, min(args.steps, 3)), interleaved=True)
        line["b128"] = run_b32(mtp, stream, 1, 1, batch=128)
    if not args.no_sweep:
        line["sweep"] = run_sweep(mtp, stream)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def run_profile_b32():
    """A small batch-32 decode for kernel captures (not a measurement): 32 slots with
    40-position prompts (one prefill chunk each), then PROFILE_B32_STEPS decode steps.
    Per prefill chunk the batched path launches 48 GEMMs and 12 attention kernels;
    per decode step 49 GEMMs (the heads' included) and 12 attention kernels."""
    import torch
    from paper_2410_13839_gb300 import build
    build.build()
    from paper_2410_13839_gb300 import mtp
    w = synth.make_weights(MODEL)
    stream = torch.cuda.Stream()
    dec = mtp.MTPDecoder(MODEL, w, synth.weight_names(MODEL), synth.is_matrix, B32, 512, stream=stream)
    for b in range(B32):
        ph, ac = synth.make_prompt(100 + b, 10, 30, MODEL.phone_vocab)
        dec.prefill(b, ph, ac, 400)
    for _ in range(PROFILE_B32_STEPS):
        mtp.mtp_decode_step(dec.ctx, N_HEADS, TOP_K)
    torch.cuda.synchronize()
    dec.close()
    print(json.dumps({"profile_b32": "done", "slots": B32, "decode_steps": PROFILE_B32_STEPS}), flush=True)


PROFILE_B32_STEPS = 12


def run_profile_b32_serving():
    """Kernel captures at serving context lengths (not a measurement): the 32 batched-serving
    prompts admitted and prefilled together (mtp_prefill_pending), then
    PROFILE_SERVING_STEPS decode steps, so the contexts reach ~1,200 keys.  Prints how many
    attention launches (attn_kernel) ran before the last step: a capture of the last step's
    first attention skips that many."""
    import torch
    from paper_2410_13839_gb300 import build
    build.build()
    from paper_2410_13839_gb300 import mtp
    seqs = b32_sequences(B32)
    max_ctx = max(len(p) + len(a) + g for p, a, g in seqs) + MODEL.n_heads_max + 8
    w = synth.make_weights(MODEL)
    stream = torch.cuda.Stream()
    dec = mtp.MTPDecoder(MODEL, w, synth.weight_names(MODEL), synth.is_matrix, B32, max_ctx, stream=stream)
    for b, (p, a, g) in enumerate(seqs):
        mtp.mtp_admit(dec.ctx, b, p, a, g)
    passes = mtp.mtp_prefill_pending(dec.ctx)
    for _ in range(PROFILE_SERVING_STEPS):
        mtp.mtp_decode_step(dec.ctx, N_HEADS, TOP_K)
    torch.cuda.synchronize()
    dec.close()
    before_last = (passes + PROFILE_SERVING_STEPS - 1) * MODEL.layers
    print(json.dumps({"profile_b32_serving": "done", "prefill_passes": passes, "decode_steps": PROFILE_SERVING_STEPS,
                      "attention_launches_before_last_step": before_last}), flush=True)


PROFILE_SERVING_STEPS = 200


def run_profile_select():
    """Kernel captures of the selection kernels (not a measurement): three mtp_viterbi
    calls on the C5 lattices (10^4 x 8 x 16), then four B=1 decode steps of the
    VALL-E-sized model (prompt 64 + 225, n=4, top_k=4), each one select_kernel launch."""
    import torch
    from paper_2410_13839_gb300 import build
    build.build()
    from paper_2410_13839_gb300 import mtp
    V = MODEL.codec_vocab
    c_ids, c_lp = c5_lattices(C5_LATTICES, C5_N, C5_K, V)
    t_ids, t_lp = torch.from_numpy(c_ids).cuda(), torch.from_numpy(c_lp).cuda()
    t_q = torch.from_numpy(synth.transition_log_q(V)).cuda()
    path = torch.zeros((C5_LATTICES, C5_N), dtype=torch.int32, device="cuda")
    acc = torch.zeros(C5_LATTICES, dtype=torch.int32, device="cuda")
    s = torch.cuda.current_stream()
    for _ in range(3):
        mtp.mtp_viterbi(C5_LATTICES, C5_N, C5_K, V, MODEL.eos_id, t_ids, t_lp, t_q, None, path, None, acc, None, s)
    torch.cuda.synchronize()
    w = synth.make_weights(MODEL)
    dec = mtp.MTPDecoder(MODEL, w, synth.weight_names(MODEL), synth.is_matrix, 1, 1100)
    try:
        ph, ac = synth.make_prompt(0, 64, 225, MODEL.phone_vocab)
        dec.prefill(0, ph, ac, 750)
        for _ in range(4):
            dec.decode_step(4, 4)
        torch.cuda.synchronize()
    finally:
        dec.close()
    print(json.dumps({"profile_select": "done", "viterbi_calls": 3, "decode_steps": 4}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--oracle-rate-steps", type=int, default=0, help=argparse.SUPPRESS)  # child of cpu_baseline
    ap.add_argument("--no-b32", action="store_true", help="skip the batch-32 serving measurement")
    ap.add_argument("--no-sweep", action="store_true", help="skip the head/beam sweep")
    ap.add_argument("--no-c5", action="store_true", help="skip the isolated heads + Viterbi microbenchmark")
    ap.add_argument("--profile-b32", action="store_true",
                    help="only run a small batch-32 decode for kernel captures (prints no measurement)")
    ap.add_argument("--profile-b32-serving", action="store_true",
                    help="only run the batch-32 serving prompts and 200 decode steps for captures (no measurement)")
    ap.add_argument("--profile-select", action="store_true",
                    help="only run the Viterbi and selection kernels for captures (prints no measurement)")
    args = ap.parse_args()
    if args.oracle_rate_steps:
        value, sample = _oracle_rate(args.oracle_rate_steps)
        print(json.dumps({"value": value, "sample": sample}), flush=True)
    elif args.profile_b32:
        run_profile_b32()
    elif args.profile_b32_serving:
        run_profile_b32_serving()
    elif args.profile_select:
        run_profile_select()
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()

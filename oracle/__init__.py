"""CPU oracle of the MTP decode hot path -- TEST INFRASTRUCTURE, not product code.

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
arm may import anything under oracle/.  The CUDA path never calls it and
shares no code with it; both sides only read the seeded inputs of `synth`.

Arithmetic: model step in float64 (numpy), with the weights upcast from their
stored fp32/bf16 values.  Every integer decision (top-k membership and order,
Viterbi path, accepted count) is taken on float32 scores, the precision the
CUDA kernels decide in.

Modules:
  model.py   -- the AR decoder of Eq. (1): one concatenated sequence
                (Sec. III-A), pre-LN blocks, KV cache, final LayerNorm.
  select.py  -- n MTP heads (Sec. III-B), log-softmax, top-k, Viterbi over the
                candidate lattice (Sec. III-C) and its decision margin.
  mtp.py     -- the multi-token inference loop (Fig. 1 caption, Sec. III-B):
                prefill, step, generate, acceptance.

Parity status per function is stated in each module header.
"""

"""fp64 CPU oracle for the artifact-KV read path (test infrastructure only).

This package is test infrastructure.  Only the tests, the smoke check in
``__graft_entry__.smoke()`` and the ``cpu_baseline`` / reference leg of
``bench.py`` may import it.  The product path (the CUDA library and its
Python binding) never imports, links or executes anything here, and the
oracle shares no code with that path.

Every function is a plain restatement of the paper's definitions in float64:
  * Sec. 3, Eq. (query-adaptation): q~ = W^Q h + (alpha/r) B A h, then the
    model's original query normalisation and RoPE;
  * Sec. 2, Eq. (1) and Eq. (full-vs-pic): artifacts cached independently and
    assembled in prompt order;
  * Sec. 2.2, Eq. (routing-oracle): softmax(q K^T / sqrt(d_k) + M_t) V, and
    the combination of its value over parts of the key set (split-KV);
  * App. A.5 (Deployment): merged W^Q + (alpha/r) B A, SDPA with causal masks
    and position ids for the assembled context;
  * the suffix tokens' own keys and values: base k_proj / v_proj (the
    adaptation touches W^Q only, Sec. 3), key normalisation and RoPE at their
    assembled positions;
  * prompt layouts whose online text (instructions, separators, the question)
    interleaves with the cached artifact spans (App. prompt construction);
  * two variants of the read from the paper's training-free baselines
    (App. C.2): keys stored before RoPE and rotated to their assembled
    positions at assembly (EPIC), and separate attention over the cached
    context (temperature T) and the online tokens combined by calibrated
    log-sum-exp terms (APE).

Parity status: every function is pinned by the tests in
``tests/test_oracle_pins.py`` (closed forms, hand-derived fixtures under
``tests/golden/``, invariants and an fp64 SDPA library cross-check).  The
rotary convention (rotate-half pairing, theta = 1e6) and the RMSNorm epsilon
are readings where the paper is silent; they are pinned to their stated
definition, not to the paper.
"""

from .attuner_oracle import (  # noqa: F401
    bf16_to_f64,
    lora_q_projection,
    merged_q_weight,
    rms_norm_heads,
    rope_rotate_half,
    query_positions,
    kv_projection,
    assemble,
    attention,
    merge_partials,
    request_forward,
    layout_online_positions,
    layout_forward,
    rotate_at_assembly,
    epic_request_forward,
    ape_combine,
    ape_request_forward,
    workload_reference,
)

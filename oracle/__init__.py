"""fp64 CPU oracle for the OLIVE per-token path (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
and reference legs may import this package.
"""
from .olive_oracle import (  # noqa: F401
    OracleError,
    bf16_bits_to_f64,
    log_softmax_rows,
    logits,
    splice_pack,
    token_divergence,
    token_logprob,
    token_topk,
    token_topk_compare,
    token_topk_kl_bwd,
    token_loss_bwd,
    token_loss_bwd_rows,
    token_loss_bwd_vocab,
)

"""olive_token_logprob_fwd_noalloc against olive_token_logprob_fwd.

The no-allocation variant exists for callers that cannot give the library a
workspace (a plugin inside a framework whose allocator owns all device memory,
or code that must not call cudaMalloc).  It takes its scratch from one device
array built into the library.  Here it is called through the C ABI twice in a
row, on two different batches, and each result must match the regular
workspace-based call within the parity tolerances; the second call also shows
that what the first left in the shared array does not leak into it.  The file
is named so that pytest collects it last.
"""

import numpy as np
import pytest
import torch

from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import assert_close_logp, assert_close_loss, gpu_pack

pytestmark = pytest.mark.gpu


def _both(b, h, W, inv_tau, reduction):
    g = gpu_pack(b)
    hc, Wc = h.cuda(), W.cuda()
    st_ref, st_na = B.new_status(), B.new_status()
    ref = B.olive_token_logprob_fwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], inv_tau, reduction,
                                    dev_status=st_ref)
    got = B.olive_token_logprob_fwd_noalloc(hc, Wc, g["targets"], g["rows"], g["n_rows"], inv_tau,
                                            reduction, dev_status=st_na)
    torch.cuda.synchronize()
    assert B.status_bits(st_ref) == [] and B.status_bits(st_na) == []
    return [t.cpu().numpy() for t in ref], [t.cpu().numpy() for t in got]


def test_noalloc_matches_workspace_call_twice():
    cases = [
        # larger batch first, so the second call runs over stale contents
        (synth.random_case(77, 16, 32000, 2048, max_prefix=60, max_cont=120, std_w=0.03), 1.0, "sum"),
        ((synth.make_batch("tiny"), synth.make_hidden("tiny", synth.make_batch("tiny").T),
          synth.make_weight("tiny")), 0.9, "mean"),
    ]
    for (b, h, W), inv_tau, red in cases:
        (rl, rs, rloss), (gl, gs, gloss) = _both(b, h, W, inv_tau, red)
        assert_close_logp(gl, rl, "logp")
        assert_close_logp(gs, rs, "lse")
        assert_close_loss(gloss[0], rloss[0])
        assert np.array_equal(gl == 0, rl == 0)


def test_noalloc_rejects_sizes_beyond_the_array():
    T, d, V = 8192, 4096, 1000
    assert B.olive_workspace_size("logprob_fwd", T, d, V) > 32 * 1024 * 1024
    h = torch.zeros(T, d, dtype=torch.bfloat16, device="cuda")
    W = torch.zeros(V, d, dtype=torch.bfloat16, device="cuda")
    i = torch.zeros(T, dtype=torch.int32, device="cuda")
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(B.OliveError) as e:
        B.olive_token_logprob_fwd_noalloc(h, W, i, i, n)
    assert e.value.status == 2  # OLIVE_ERR_SHAPE, returned before any launch

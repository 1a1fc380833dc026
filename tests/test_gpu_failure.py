"""Failure detection without a GPU fault: a host-set test hook
(archer_debug_stall_attention) makes the attention kernel withhold its last
P V product, so the softmax warps' bounded
wait expires (in both kernel instantiations).  The kernel must leave cleanly (TMEM freed, no trap, no hang),
archer_check_device must report ARCHER_ERR_TIMEOUT, and the context must stay
usable: the next call is correct."""
import math

import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_08086_gb300 import synth

pytestmark = pytest.mark.gpu


# (B, G, H): G = 256 with two heads takes one tile per CTA (a small grid):
# the one-tile kernel (S double buffered); 40 heads x 2 tile pairs = 80 pairs
# (more than half the SMs): the two-tile kernel; B 8 x 8 heads x 10 tile pairs
# = 640 work items (four per SM or more): the persistent two-tile kernel,
# whose abort path also ends the walk over its items.
@pytest.mark.parametrize("B,G,H", [(1, 256, 2), (1, 512, 40), (8, 2560, 8)],
                         ids=["one-tile", "two-tile", "persistent"])
def test_expired_wait_reports_timeout_and_context_survives(B, G, H):
    from paper_2608_08086_gb300 import archer as A
    P, D = 128, 64
    bits = synth.attn_inputs(synth.AttnShape(B, P, G, H, H, D), seed=9)
    d = {k: torch.from_numpy(v.view(np.int16)).view(torch.bfloat16).cuda() for k, v in bits.items()}
    shape = A.make_shape(B, P, G, H, H, D)
    q = d["q_all"][:, P:].contiguous()
    out = torch.zeros(B, G, H, D, dtype=torch.bfloat16, device="cuda")
    A.archer_check_device()                                  # start from a clean error word
    assert not A.archer_debug_stall_attention(True)
    try:
        A.archer_attn_step(shape, q, d["k_cache"], d["v_cache"], d["k_resp"], d["v_resp"], out)
    finally:
        assert A.archer_debug_stall_attention(False)
    with pytest.raises(A.ArcherError) as e:
        A.archer_check_device()
    assert e.value.status == A.ARCHER_ERR_TIMEOUT
    A.archer_check_device()                                  # the word was cleared
    A.archer_attn_step(shape, q, d["k_cache"], d["v_cache"], d["k_resp"], d["v_resp"], out)
    A.archer_check_device()
    x = {k: synth.bf16_bits_to_f64(v)[:1] for k, v in bits.items()}           # sequence 0 against the oracle
    ref, _ = O.attn_step(x["q_all"][:, P:], x["k_cache"], x["v_cache"], x["k_resp"], x["v_resp"], 1 / math.sqrt(D))
    got = synth.bf16_bits_to_f64(out[:1].contiguous().view(torch.int16).cpu().numpy().view(np.uint16))
    assert (np.abs(got - ref) <= 2e-2 + 2e-2 * np.abs(ref)).all()

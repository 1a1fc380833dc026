"""The staleness curve measured with the CUDA kernels: the cached step against
K_p(g_r) and the fresh one against K_p(g_t) (both caches rounded to bf16, as a
model would store them), compared with the oracle on the same bf16 inputs, and
below Eq. theory-radius-bound's Gamma sqrt(D_t) plus the bf16 output rounding."""
import math

import numpy as np
import pytest
import torch

from oracle import oracle as O
from oracle import staleness as S
from paper_2608_08086_gb300 import synth

pytestmark = pytest.mark.gpu


def _dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def test_staleness_curve_on_gpu_matches_oracle_and_bound():
    from paper_2608_08086_gb300 import archer as A
    shape = synth.AttnShape(2, 200, 72, 4, 2, 64)
    B, P, G, Hq, Hkv, D = 2, 200, 72, 4, 2, 64
    m = synth.staleness_model(shape, seed=5)
    scale = 1.0 / math.sqrt(D)
    g_r = synth.staleness_tokens(5, B, G)
    kc, vc = synth.staleness_prompt_cache(m, g_r, Hkv, D)
    kc_b, vc_b = synth.to_bf16_bits(kc), synth.to_bf16_bits(vc)
    q, kg, vg = m["q_resp"], m["k_resp"], m["v_resp"]
    sh = A.make_shape(B, P, G, Hq, Hkv, D)
    dq, dkg, dvg = _dev(q), _dev(kg), _dev(vg)
    f64 = synth.bf16_bits_to_f64
    gam = S.gamma(m, f64(q), f64(vc_b), f64(vg), scale)

    def run(kb, vb):
        out = torch.empty(B, G, Hq, D, dtype=torch.bfloat16, device="cuda")
        A.archer_attn_step(sh, dq, _dev(kb), _dev(vb), dkg, dvg, out)
        return f64(out.view(torch.int16).cpu().numpy().view(np.uint16))

    o_cached = run(kc_b, vc_b)
    r_cached, _ = O.attn_step(f64(q), f64(kc_b), f64(vc_b), f64(kg), f64(vg), scale)
    prev = 0.0
    for d in (0, 1, 4, 16, 72):
        kf, vf = synth.staleness_prompt_cache(m, synth.staleness_drift(g_r, d, 5), Hkv, D)
        kf_b, vf_b = synth.to_bf16_bits(kf), synth.to_bf16_bits(vf)
        o_fresh = run(kf_b, vf_b)
        r_fresh, _ = O.attn_step(f64(q), f64(kf_b), f64(vf_b), f64(kg), f64(vg), scale)
        err_gpu = np.abs(o_cached - o_fresh).max()
        err_ref = np.abs(r_cached - r_fresh).max()
        # two bf16-rounded outputs: at most one output ulp each, plus fp32 accumulation
        slack = 2 * 2.0 ** -8 * max(np.abs(r_cached).max(), np.abs(r_fresh).max())
        assert abs(err_gpu - err_ref) <= slack, (d, err_gpu, err_ref)
        assert err_gpu <= gam * math.sqrt(d) + slack, (d, err_gpu, gam * math.sqrt(d))
        if d == 0:
            assert err_gpu == 0.0
        prev = max(prev, err_ref)
    assert prev > 0

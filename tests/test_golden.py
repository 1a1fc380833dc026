"""Hand-derived fixtures under tests/golden/, checked against the fp64 oracle
(CPU) and against the CUDA path through the C ABI (GPU).

The fixtures are worked by hand from the definitions (each file states its
passage and each case its derivation): attention weights that are small
rationals (Sec. 4.1, Eq. archer-attention; refresh of Sec. 4.2), decoder scores
of short logit rows (Sec. 6, Eq. theory-margin), and refresh decisions of the
state-anchored rule (Eq. archer-distance, Eq. archer-controller, the age signal
of Sec. 6).  No value in them comes from either implementation.
"""
import json
import math
import os

import numpy as np
import pytest

from oracle import oracle as O

HERE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
ORACLE_TOL = 1e-12
ATOL = RTOL = 2e-2            # attention on bf16 inputs, as in the parity tests
P_ATOL, P_RTOL = 1e-5, 1e-4   # probabilities from fp32 logits


def _load(name):
    with open(os.path.join(HERE, name)) as f:
        return json.load(f)["cases"]


ATTN = _load("attention_closed_form.json")
SCORES = _load("decode_scores_closed_form.json")
RULE = _load("refresh_rule_cases.json")


def _arr(x, shape):
    return np.asarray(x, dtype=np.float64).reshape(shape)


def _attn_case(c):
    B, P, G, Hq, Hkv, D = 1, c["P"], c["G"], c["Hq"], c["Hkv"], c["D"]
    t = {
        "q_all": _arr(c["q_all"], (B, P + G, Hq, D)),
        "k_cache": _arr(c["k_cache"], (B, P, Hkv, D)), "v_cache": _arr(c["v_cache"], (B, P, Hkv, D)),
        "k_new": _arr(c["k_new"], (B, P, Hkv, D)), "v_new": _arr(c["v_new"], (B, P, Hkv, D)),
        "k_resp": _arr(c["k_resp"], (B, G, Hkv, D)), "v_resp": _arr(c["v_resp"], (B, G, Hkv, D)),
        "out_step": _arr(c["out_step"], (B, G, Hq, D)), "out_refresh": _arr(c["out_refresh"], (B, P + G, Hq, D)),
    }
    return (B, P, G, Hq, Hkv, D), t


def _logits(c):
    return np.array([-math.inf if v == "-inf" else float(v) for v in c["z"]], dtype=np.float64)


# ----------------------------------------------------------------------------- oracle (CPU)

@pytest.mark.parametrize("c", ATTN, ids=[c["name"] for c in ATTN])
def test_oracle_attention_golden(c):
    (B, P, G, Hq, Hkv, D), t = _attn_case(c)
    out_s, _ = O.attn_step(t["q_all"][:, P:], t["k_cache"], t["v_cache"], t["k_resp"], t["v_resp"], c["scale"])
    np.testing.assert_allclose(out_s, t["out_step"], rtol=0, atol=ORACLE_TOL)
    out_r, _, kc, vc = O.prompt_refresh(t["q_all"], t["k_new"], t["v_new"], t["k_resp"], t["v_resp"],
                                        t["k_cache"], t["v_cache"], c["scale"])
    np.testing.assert_allclose(out_r, t["out_refresh"], rtol=0, atol=ORACLE_TOL)
    assert np.array_equal(kc, t["k_new"]) and np.array_equal(vc, t["v_new"]), "refresh rewrites the cache"


@pytest.mark.parametrize("c", SCORES, ids=[c["name"] for c in SCORES])
def test_oracle_scores_golden(c):
    z = _logits(c)[None, :]
    r = O.decode_scores(z, mask_state=np.array([1 if c["masked"] else 0], dtype=np.uint8),
                        cur_tokens=np.array([c["cur"]], dtype=np.int32))
    assert int(r["top1"][0]) == c["top1"]
    for k in ("max_prob", "margin", "cur_prob"):
        assert abs(r[k][0] - c[k]) <= ORACLE_TOL, k


@pytest.mark.parametrize("c", RULE, ids=[c["why"] for c in RULE])
def test_oracle_rule_golden(c):
    dist, flag, ga, ag = O.should_refresh(np.array([c["cur"]], dtype=np.int32), np.array([c["anchor"]], dtype=np.int32),
                                          np.array([c["age"]], dtype=np.int32), c["K"], c["max_age"])
    assert (int(dist[0]), int(flag[0]), int(ag[0])) == (c["dist"], c["flag"], c["age_out"])
    assert ga[0].tolist() == c["anchor_out"]


# ----------------------------------------------------------------------------- CUDA path (GPU)

@pytest.fixture(scope="module")
def A():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2608_08086_gb300 import archer
    return archer


def _dev_bf16_padded(x, D):
    """[.., d] fp64 -> [.., D] bf16 on the GPU, zero-padded (dot products and
    the first d output columns are unchanged)."""
    import torch
    pad = np.zeros(x.shape[:-1] + (D,))
    pad[..., : x.shape[-1]] = x
    return torch.from_numpy(pad).to(torch.bfloat16).cuda()


def _check_attn(got, ref, what):
    g = got.float().cpu().numpy().astype(np.float64)
    d = ref.shape[-1]
    assert np.all(g[..., d:] == 0), f"{what}: padded columns must stay 0"
    err = np.abs(g[..., :d] - ref) - (ATOL + RTOL * np.abs(ref))
    assert (err <= 0).all(), f"{what}: max excess {err.max():.3g}\n{g[..., :d]}\nvs\n{ref}"


@pytest.mark.gpu
@pytest.mark.parametrize("c", ATTN, ids=[c["name"] for c in ATTN])
@pytest.mark.parametrize("Dk", [64, 128])
def test_gpu_attention_golden(A, c, Dk):
    import torch
    (B, P, G, Hq, Hkv, D), t = _attn_case(c)
    d = {k: _dev_bf16_padded(v, Dk) for k, v in t.items() if not k.startswith("out")}
    sh = A.make_shape(B, P, G, Hq, Hkv, Dk, c["scale"])
    out_s = torch.empty(B, G, Hq, Dk, dtype=torch.bfloat16, device="cuda")
    A.archer_attn_step(sh, d["q_all"][:, P:].contiguous(), d["k_cache"], d["v_cache"], d["k_resp"], d["v_resp"],
                       out_s)
    kc, vc = d["k_cache"].clone(), d["v_cache"].clone()
    out_r = torch.empty(B, P + G, Hq, Dk, dtype=torch.bfloat16, device="cuda")
    A.archer_prompt_refresh(sh, d["q_all"], d["k_new"], d["v_new"], d["k_resp"], d["v_resp"], out_r, None, kc, vc)
    A.archer_check_device()
    _check_attn(out_s, t["out_step"], "cached step")
    _check_attn(out_r, t["out_refresh"], "refresh")
    assert torch.equal(kc, d["k_new"]) and torch.equal(vc, d["v_new"]), "refresh rewrites the cache"


@pytest.mark.gpu
@pytest.mark.parametrize("c", SCORES, ids=[c["name"] for c in SCORES])
def test_gpu_scores_golden(A, c):
    import torch
    z = torch.from_numpy(_logits(c)[None, :].astype(np.float32)).cuda()
    mp = torch.empty(1, dtype=torch.float32, device="cuda")
    t1 = torch.empty(1, dtype=torch.int32, device="cuda")
    mg = torch.empty(1, dtype=torch.float32, device="cuda")
    cp = torch.empty(1, dtype=torch.float32, device="cuda")
    A.archer_decode_scores(z, mp, t1, mg, mask_state=torch.tensor([1 if c["masked"] else 0], dtype=torch.uint8,
                                                                   device="cuda"),
                           cur_tokens=torch.tensor([c["cur"]], dtype=torch.int32, device="cuda"), cur_prob=cp)
    A.archer_check_device()
    assert int(t1[0]) == c["top1"]
    for k, v in (("max_prob", mp), ("margin", mg), ("cur_prob", cp)):
        assert abs(float(v[0]) - c[k]) <= P_ATOL + P_RTOL * abs(c[k]), k


@pytest.mark.gpu
@pytest.mark.parametrize("c", RULE, ids=[c["why"] for c in RULE])
def test_gpu_rule_golden(A, c):
    import torch
    g = torch.tensor([c["cur"]], dtype=torch.int32, device="cuda")
    ga = torch.tensor([c["anchor"]], dtype=torch.int32, device="cuda")
    age = torch.tensor([c["age"]], dtype=torch.int32, device="cuda")
    dist = torch.empty(1, dtype=torch.int32, device="cuda")
    flag = torch.empty(1, dtype=torch.uint8, device="cuda")
    A.archer_should_refresh(g, ga, age, c["K"], c["max_age"], True, dist, flag)
    A.archer_check_device()
    assert (int(dist[0]), int(flag[0]), int(age[0])) == (c["dist"], c["flag"], c["age_out"])
    assert ga[0].tolist() == c["anchor_out"]

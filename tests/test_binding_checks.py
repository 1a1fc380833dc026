"""The Python binding rejects wrong sizes before any pointer reaches the
library (the kernels and the step graph take raw addresses, so a wrong size
would otherwise read or write out of bounds on the device).  On the CPU: a
tensor of the wrong shape raises ValueError; one of the right shape raises
TypeError because it is not a CUDA tensor, so nothing is ever launched here."""
import pytest
import torch

from paper_2608_08086_gb300 import build

build.build()                     # the binding refuses to import without the library
from paper_2608_08086_gb300 import archer as A  # noqa: E402

B, P, G, Hq, Hkv, D = 2, 128, 64, 4, 2, 64
N = P + G
SHAPE = A.make_shape(B, P, G, Hq, Hkv, D)
bf = torch.bfloat16


def z(*shape, dtype=bf):
    return torch.zeros(shape, dtype=dtype)


def layer(**override):
    lay = {"q_all": z(B, N, Hq, D), "q_resp": z(B, G, Hq, D), "k_prompt_new": z(B, P, Hkv, D),
           "v_prompt_new": z(B, P, Hkv, D), "k_resp": z(B, G, Hkv, D), "v_resp": z(B, G, Hkv, D),
           "k_cache": z(B, P, Hkv, D), "v_cache": z(B, P, Hkv, D), "out_full": z(B, N, Hq, D),
           "out_step": z(B, G, Hq, D)}
    lay.update(override)
    return lay


def step_graph(layers, **kw):
    i32 = torch.int32
    args = dict(g_cur=z(B, G, dtype=i32), g_anchor=z(B, G, dtype=i32), age=z(B, dtype=i32), K=8, max_age=4,
                flag_out=z(B, dtype=torch.uint8), dist_out=z(B, dtype=i32), refresh_count=z(1, dtype=i32))
    args.update(kw)
    return A.StepGraph(SHAPE, layers, **args)


def test_attention_calls_check_every_shape():
    good = dict(q_resp=z(B, G, Hq, D), k_cache=z(B, P, Hkv, D), v_cache=z(B, P, Hkv, D), k_resp=z(B, G, Hkv, D),
                v_resp=z(B, G, Hkv, D), out=z(B, G, Hq, D))
    for name, bad in (("q_resp", z(B, G, Hq + 1, D)), ("k_cache", z(B, P - 1, Hkv, D)), ("out", z(B, N, Hq, D)),
                      ("v_resp", z(B, G, Hkv, D // 2))):
        with pytest.raises(ValueError, match=name):
            A.archer_attn_step(SHAPE, **dict(good, **{name: bad}))
    with pytest.raises(ValueError, match="lse"):
        A.archer_attn_step(SHAPE, **good, lse=z(B, Hq, N, dtype=torch.float32))
    with pytest.raises(TypeError, match="CUDA"):
        A.archer_attn_step(SHAPE, **good, workspace=False)
    with pytest.raises(ValueError, match="refresh_flags"):
        A.archer_prompt_refresh(SHAPE, z(B, N, Hq, D), z(B, P, Hkv, D), z(B, P, Hkv, D), z(B, G, Hkv, D),
                                z(B, G, Hkv, D), z(B, N, Hq, D), refresh_flags=z(B + 1, dtype=torch.uint8),
                                workspace=False)


def test_step_graph_checks_every_layer_and_output_before_capture():
    for name, bad in (("q_all", z(B, G, Hq, D)), ("k_cache", z(B, P, Hq, D)), ("out_step", z(B, N, Hq, D)),
                      ("v_prompt_new", z(B, P + 1, Hkv, D))):
        with pytest.raises(ValueError, match=name):
            step_graph([layer(), layer(**{name: bad})])
    with pytest.raises(ValueError, match="g_anchor"):
        step_graph([layer()], g_anchor=z(B, G + 1, dtype=torch.int32))
    with pytest.raises(ValueError, match="dist_out"):
        step_graph([layer()], dist_out=z(B + 1, dtype=torch.int32))
    rows = B * G
    with pytest.raises(ValueError, match="margin"):
        step_graph([layer()], logits=z(rows, 100), max_prob=z(rows, dtype=torch.float32),
                   top1=z(rows, dtype=torch.int32), margin=z(rows - 1, dtype=torch.float32))
    # every size right: the first pointer marshalled refuses a CPU tensor
    with pytest.raises(TypeError, match="CUDA"):
        step_graph([layer(), layer()])


def test_scoring_and_rewrite_check_sizes():
    rows = B * G
    outs = dict(max_prob=z(rows, dtype=torch.float32), top1=z(rows, dtype=torch.int32),
                margin=z(rows, dtype=torch.float32))
    with pytest.raises(ValueError, match="mask_state"):
        A.archer_decode_scores(z(B, G, 100), **outs, mask_state=z(rows + 1, dtype=torch.uint8), workspace=z(16))
    with pytest.raises(ValueError, match="cur_tokens"):
        A.archer_decode_scores(z(B, G, 100), **outs, cur_tokens=z(rows - 1, dtype=torch.int32), workspace=z(16))
    with pytest.raises(ValueError, match="top1"):
        A.archer_decode_scores(z(B, G, 100), **dict(outs, top1=z(rows, dtype=torch.int64)), workspace=z(16))
    with pytest.raises(ValueError, match="k_dst"):
        A.archer_cache_rewrite(SHAPE, z(B, P, Hkv, D), None, z(B, P, Hkv, D + 1), None)
    with pytest.raises(ValueError, match="refresh_flags"):
        A.archer_cache_rewrite(SHAPE, z(B, P, Hkv, D), None, z(B, P, Hkv, D), None,
                               refresh_flags=z(1, dtype=torch.uint8))
    with pytest.raises(ValueError, match="g_anchor"):
        A.archer_should_refresh(z(B, G, dtype=torch.int32), z(B, G - 1, dtype=torch.int32), z(B, dtype=torch.int32),
                                8, 4, True, None, z(B, dtype=torch.uint8))

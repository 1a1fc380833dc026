"""Out-of-bounds writes: every output and workspace of the C ABI is carved
out of a larger buffer whose margins hold a canary pattern; after the calls
the margins must be untouched (compute-sanitizer being closed on this pool,
this stands in for its memcheck on odd shapes: ragged tiles, G = 1, P = 0,
split launches, ragged vocabularies)."""
import numpy as np
import pytest
import torch

from paper_2608_08086_gb300 import synth

pytestmark = pytest.mark.gpu

PAD = 4096          # bytes of canary on each side (a multiple of 16 keeps the interior aligned)
CANARY = 0xA5


def guarded(shape, dtype):
    n = int(np.prod(shape)) * torch.tensor([], dtype=dtype).element_size()
    raw = torch.full((n + 2 * PAD,), CANARY, dtype=torch.uint8, device="cuda")
    inner = raw[PAD:PAD + n].view(dtype).view(*shape)
    return raw, inner


def intact(raw):
    head, tail = raw[:PAD], raw[-PAD:]
    return bool((head == CANARY).all() and (tail == CANARY).all())


def dev_bf16(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


@pytest.mark.parametrize("case", [(2, 100, 37, 8, 2, 128), (1, 0, 1, 2, 1, 64), (1, 1900, 70, 3, 1, 64),
                                  (3, 129, 130, 4, 1, 64)])
def test_attention_writes_stay_inside(case):
    from paper_2608_08086_gb300 import archer as A
    B, P, G, Hq, Hkv, D = case
    bits = synth.attn_inputs(synth.AttnShape(B, P, G, Hq, Hkv, D), seed=3)
    d = {k: dev_bf16(v) for k, v in bits.items()}
    shape = A.make_shape(B, P, G, Hq, Hkv, D)
    N = P + G
    for M, call in ((G, "step"), (N, "refresh")):
        raw_o, out = guarded((B, M, Hq, D), torch.bfloat16)
        raw_l, lse = guarded((B, Hq, M), torch.float32)
        ws_n = A.archer_attn_workspace_size(shape, M)
        raw_w, ws = guarded((max(ws_n, 16),), torch.uint8)
        if call == "step":
            A.archer_attn_step(shape, d["q_all"][:, P:].contiguous(), d["k_cache"], d["v_cache"], d["k_resp"],
                               d["v_resp"], out, lse, workspace=ws)
        else:
            raw_kc, kc = guarded((B, P, Hkv, D), torch.bfloat16)
            raw_vc, vc = guarded((B, P, Hkv, D), torch.bfloat16)
            flags = torch.tensor([1, 0, 1][:B], dtype=torch.uint8, device="cuda")
            A.archer_prompt_refresh(shape, d["q_all"], d["k_prompt"], d["v_prompt"], d["k_resp"], d["v_resp"], out,
                                    lse, kc, vc, refresh_flags=flags, workspace=ws)
            torch.cuda.synchronize()
            assert intact(raw_kc) and intact(raw_vc), f"cache rewrite {case}"
        torch.cuda.synchronize()
        A.archer_check_device()
        assert intact(raw_o), f"out {call} {case}"
        assert intact(raw_l), f"lse {call} {case}"
        assert intact(raw_w), f"workspace {call} {case}"


@pytest.mark.parametrize("rows,V,stride,dtype", [(5, 1001, 1008, torch.bfloat16), (3, 70000, 70004, torch.float32),
                                                 (2, 1, 8, torch.bfloat16)])
def test_scoring_and_rule_writes_stay_inside(rows, V, stride, dtype):
    from paper_2608_08086_gb300 import archer as A
    g = torch.Generator(device="cuda").manual_seed(1)
    z = torch.randn(rows, stride, device="cuda", generator=g).to(dtype)
    outs = {n: guarded((rows,), t) for n, t in (("mp", torch.float32), ("t1", torch.int32), ("mg", torch.float32),
                                                ("cp", torch.float32))}
    n_ws = A.archer_decode_scores_workspace_size(rows, V)
    raw_w, ws = guarded((max(n_ws, 16),), torch.uint8)
    cur = torch.zeros(rows, dtype=torch.int32, device="cuda")
    A.archer_decode_scores(z, outs["mp"][1], outs["t1"][1], outs["mg"][1], cur_tokens=cur, cur_prob=outs["cp"][1],
                           vocab=V, workspace=ws)
    torch.cuda.synchronize()
    for n, (raw, _) in outs.items():
        assert intact(raw), n
    assert intact(raw_w)
    # the refresh rule and the decoder update on a ragged resp_len
    B, G = 3, 37
    gc = torch.randint(0, 9, (B, G), dtype=torch.int32, device="cuda", generator=g)
    raw_ga, ga = guarded((B, G), torch.int32)
    ga.copy_(gc)
    raw_age, age = guarded((B,), torch.int32)
    age.zero_()
    raw_d, dist = guarded((B,), torch.int32)
    raw_f, flag = guarded((B,), torch.uint8)
    A.archer_should_refresh(gc, ga, age, 2, 3, True, dist, flag)
    raw_ch, ch = guarded((B, G), torch.uint8)
    mp = torch.rand(B * G, device="cuda", generator=g)
    A.archer_decoder_update(gc, mp, torch.zeros(B * G, dtype=torch.int32, device="cuda"), mp, ch, 0.5, 0.1)
    torch.cuda.synchronize()
    for raw in (raw_ga, raw_age, raw_d, raw_f, raw_ch):
        assert intact(raw)

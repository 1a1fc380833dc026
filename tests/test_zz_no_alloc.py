"""The allocation-free scoring entry point (archer_decode_scores_noalloc).

Callers that cannot allocate device memory (code inside another framework's
memory pool, latency-critical loops that must not synchronise on cudaMalloc,
bindings without an allocator) use this variant; its scratch is a static
device array of the library.  Checked here through the C ABI against the fp64
oracle on sampled rows and against the workspace entry point on every row, on
two calls in a row (the second reuses the scratch the first left behind),
with the scoring tolerances of the other tests.  This file is collected last
so that a failure here stops a -x run only after every other test has run."""
import ctypes

import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_08086_gb300 import synth

pytestmark = pytest.mark.gpu

SCRATCH_BYTES = 4 << 20


def _lib():
    from paper_2608_08086_gb300 import archer as A
    L = A.lib
    vp = ctypes.c_void_p
    L.archer_decode_scores_noalloc.argtypes = [ctypes.c_int] * 4 + [vp, ctypes.c_int64] + [vp] * 7
    L.archer_decode_scores_noalloc.restype = ctypes.c_int
    L.archer_last_error.restype = ctypes.c_char_p
    return A, L


def _call(fn, z, vocab, dtype_code, mask=None, cur=None, extra=()):
    rows = z.shape[0]
    mp = torch.full((rows,), -1.0, dtype=torch.float32, device="cuda")
    t1 = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
    mg = torch.full((rows,), -1.0, dtype=torch.float32, device="cuda")
    cp = torch.full((rows,), -1.0, dtype=torch.float32, device="cuda")
    p = lambda t: None if t is None else ctypes.c_void_p(t.data_ptr())  # noqa: E731
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = fn(1, rows, vocab, dtype_code, p(z), ctypes.c_int64(z.shape[1]), p(mask), p(cur), p(mp), p(t1), p(mg),
            p(cp), *extra, stream)
    torch.cuda.synchronize()
    return rc, {"max_prob": mp.cpu().numpy().astype(np.float64), "top1": t1.cpu().numpy(),
                "margin": mg.cpu().numpy().astype(np.float64), "cur_prob": cp.cpu().numpy().astype(np.float64)}


def _close(got, ref, what):
    keep = ref["margin"] >= 1e-4
    assert (got["top1"][keep] == ref["top1"][keep]).all(), f"{what}: top-1"
    for k in ("max_prob", "margin", "cur_prob"):
        err = np.abs(got[k] - ref[k])
        assert (err <= 1e-5 + 1e-4 * np.abs(ref[k])).all(), f"{what}: {k} max err {err.max():.3e}"


def _host_f64(z):
    if z.dtype == torch.bfloat16:
        return synth.bf16_bits_to_f64(z.contiguous().view(torch.int16).cpu().numpy().view(np.uint16))
    return z.double().cpu().numpy()


@pytest.mark.parametrize("rows,vocab,dtype", [
    (1024, 152064, "bf16"),     # ten 32 KB chunks per row
    (300, 70001, "f32"),        # nine chunks, a ragged last one
    (14000, 152064, "bf16"),    # 2.2 MB of partials: inside the scratch for bf16 (fp32 would need 4.3 MB)
])
def test_noalloc_scoring_matches_oracle_and_workspace_entry_point_twice(rows, vocab, dtype):
    A, L = _lib()
    tdt, code = (torch.bfloat16, A.ARCHER_DTYPE_BF16) if dtype == "bf16" else (torch.float32, A.ARCHER_DTYPE_F32)
    z = synth.device_logits(rows, vocab, "cuda", seed=rows, std=2.5, boost_max=6.0, dtype=tdt)
    cur = (torch.arange(rows, dtype=torch.int64, device="cuda") * 7919 % vocab).to(torch.int32)
    mask = (torch.arange(rows, device="cuda") % 2).to(torch.uint8)
    n_ws = A.archer_decode_scores_workspace_size(rows, vocab)
    ws = torch.zeros(n_ws, dtype=torch.uint8, device="cuda")
    rc, with_ws = _call(L.archer_decode_scores, z, vocab, code, mask, cur,
                        extra=(ctypes.c_void_p(ws.data_ptr()), ctypes.c_size_t(n_ws)))
    assert rc == 0, L.archer_last_error().decode()
    del ws
    sample = np.unique(np.concatenate([[0, rows - 1], np.random.default_rng(rows).integers(0, rows, 62)]))
    ref = O.decode_scores(_host_f64(z[torch.from_numpy(sample).cuda()]),
                          mask_state=mask.cpu().numpy()[sample], cur_tokens=cur.cpu().numpy()[sample])
    for call in range(2):                        # two calls in a row share the static scratch
        rc, got = _call(L.archer_decode_scores_noalloc, z, vocab, code, mask, cur)
        assert rc == 0, L.archer_last_error().decode()
        _close({k: v[sample] for k, v in got.items()}, ref, f"call {call} vs oracle")
        _close(got, with_ws, f"call {call} vs the workspace entry point")


def test_noalloc_scoring_rejects_sizes_beyond_its_scratch():
    A, L = _lib()
    z = torch.zeros(16, 8, dtype=torch.bfloat16, device="cuda")
    p = ctypes.c_void_p(z.data_ptr())
    # (rows, vocab, dtype, partial bytes): each above the 4 MiB scratch, rejected before any launch
    for rows, vocab, code, need in ((30000, 152064, A.ARCHER_DTYPE_BF16, 30000 * 10 * 16),
                                    (14000, 152064, A.ARCHER_DTYPE_F32, 14000 * 19 * 16)):
        assert need > SCRATCH_BYTES
        rc = L.archer_decode_scores_noalloc(1, rows, vocab, code, p, ctypes.c_int64(vocab), None, None, p, p, p,
                                            None, None)
        assert rc == A.ARCHER_ERR_UNSUPPORTED
        assert b"scratch" in L.archer_last_error()

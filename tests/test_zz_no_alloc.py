"""The allocation-free scoring entry point (archer_decode_scores_noalloc).

Callers that cannot allocate device memory (code inside another framework's
memory pool, latency-critical loops that must not synchronise on cudaMalloc,
bindings without an allocator) use this variant; its scratch is a static
device array of the library.  Checked here through the C ABI against the
workspace entry point, on two calls in a row (the second reuses the scratch
the first left behind), with the scoring tolerances of the other tests.
This file is collected last so that a failure here stops a -x run only after
every other test has run."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_08086_gb300 import synth

pytestmark = pytest.mark.gpu


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
    return rc, {"max_prob": mp.cpu().numpy(), "top1": t1.cpu().numpy(), "margin": mg.cpu().numpy(),
                "cur_prob": cp.cpu().numpy()}


def _close(got, ref):
    keep = ref["margin"] >= 1e-4
    assert (got["top1"][keep] == ref["top1"][keep]).all()
    for k in ("max_prob", "margin", "cur_prob"):
        assert (np.abs(got[k] - ref[k]) <= 1e-5 + 1e-4 * np.abs(ref[k])).all(), k


def test_noalloc_scoring_matches_workspace_entry_point_twice():
    from paper_2608_08086_gb300 import archer as A
    L = A.lib
    vp = ctypes.c_void_p
    L.archer_decode_scores_noalloc.argtypes = [ctypes.c_int] * 4 + [vp, ctypes.c_int64] + [vp] * 7
    L.archer_decode_scores_noalloc.restype = ctypes.c_int
    noalloc = L.archer_decode_scores_noalloc
    with_ws = L.archer_decode_scores

    cases = [
        # (rows, vocab, dtype): several chunks per row, so the scratch is used
        (1024, 152064, torch.bfloat16, A.ARCHER_DTYPE_BF16),
        (300, 70001, torch.float32, A.ARCHER_DTYPE_F32),
    ]
    for rows, vocab, tdt, code in cases:
        z = synth.device_logits(rows, vocab, "cuda", seed=rows, std=2.5, boost_max=6.0, dtype=tdt)
        cur = torch.arange(rows, dtype=torch.int32, device="cuda") * 7 % vocab
        mask = (torch.arange(rows, device="cuda") % 2).to(torch.uint8)
        n_ws = A.archer_decode_scores_workspace_size(rows, vocab)
        ws = torch.zeros(n_ws, dtype=torch.uint8, device="cuda")
        rc, ref = _call(with_ws, z, vocab, code, mask, cur, extra=(ctypes.c_void_p(ws.data_ptr()),
                                                                    ctypes.c_size_t(n_ws)))
        assert rc == 0
        for _ in range(2):                       # two calls in a row share the static scratch
            rc, got = _call(noalloc, z, vocab, code, mask, cur)
            assert rc == 0, A.lib.archer_last_error().decode()
            _close(got, ref)


def test_noalloc_scoring_rejects_sizes_beyond_its_scratch():
    from paper_2608_08086_gb300 import archer as A
    L = A.lib
    L.archer_last_error.restype = ctypes.c_char_p
    z = torch.zeros(16, 8, dtype=torch.bfloat16, device="cuda")
    p = ctypes.c_void_p(z.data_ptr())
    # 20000 rows x 152064 logits need about 6 MB of scratch: rejected before any launch
    rc = L.archer_decode_scores_noalloc(1, 20000, 152064, A.ARCHER_DTYPE_BF16, p, ctypes.c_int64(152064), None,
                                        None, p, p, p, None, None)
    assert rc == A.ARCHER_ERR_UNSUPPORTED
    assert b"scratch" in L.archer_last_error()

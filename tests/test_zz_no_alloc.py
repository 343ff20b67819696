"""The workspace-free confidence statistics (sdd_confidence_noalloc).

Some callers cannot allocate device memory where they need the statistics:
code running under CUDA stream capture, where cudaMalloc is not allowed, or a
framework whose device memory is a fixed arena it owns.  The library serves
them from a fixed scratch array of its own.  This test calls that entry point
through the C ABI twice in a row (the second call starts from whatever the
first left in the shared scratch) and checks each result against the fp64
oracle, element by element, and against sdd_confidence, which takes a
caller-provided workspace, with the tolerances of the other parity tests.  It lives in a file of its own that is collected
last, and passes both alone in a fresh process and after the other tests."""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

RTOL = {torch.bfloat16: 2e-3, torch.float32: 1e-5}
ATOL = 1e-7


def _padded(z, stride):
    B, P, V = z.shape
    buf = torch.full((B, P, stride), float("inf"), dtype=z.dtype, device=z.device)
    buf[..., :V] = z
    return buf[..., :V]


def _same(name, got, want, dtype):
    g = got.double().cpu().numpy()
    w = want.double().cpu().numpy() if isinstance(want, torch.Tensor) else np.asarray(want, np.float64)
    if name == "logq":      # a log-probability: absolute error = relative error of q
        ok = np.abs(g - w) <= RTOL[dtype]
    else:
        ok = np.abs(g - w) <= RTOL[dtype] * np.abs(w) + ATOL
    ok |= np.isnan(g) & np.isnan(w)
    assert ok.all(), f"{name}: {(~ok).sum()} entries differ"


def test_noalloc_matches_oracle_and_workspace_call_twice_in_a_row(orc):
    import paper_2608_14787_gb300 as sdd
    from paper_2608_14787_gb300 import synth
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sdd.load()
    cases = [("c3", 16, 32, 151_936, torch.bfloat16), ("tiny", 5, 9, 30_011, torch.float32)]
    for rnd, (wl, B, gamma, V, dtype) in enumerate(cases):
        blk = synth.make_block(wl, device="cuda", round_=rnd, B=B, gamma=gamma, V=V, dtype=dtype)
        esz = 2 if dtype == torch.bfloat16 else 4
        stride = -(-V * esz // 16) * 16 // esz
        z = _padded(blk.z_d, stride) if stride != V else blk.z_d
        want = sdd.confidence(z, blk.x)
        status = sdd.new_status()
        got = sdd.confidence_noalloc(z, blk.x, status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        st = orc.row_stats(synth.bf16_bits(blk.z_d), tokens=blk.x.cpu().numpy())
        for f in ("q", "logq", "maxprob", "lse", "entropy"):
            _same(f, getattr(got, f), getattr(st, f), dtype)
            _same(f, getattr(got, f), getattr(want, f), dtype)
        np.testing.assert_array_equal(got.argmax.cpu().numpy(), st.argmax)
        assert torch.equal(got.argmax, want.argmax)


def test_noalloc_rejects_batches_beyond_its_scratch():
    import paper_2608_14787_gb300 as sdd
    lib = sdd.load()
    VP = ctypes.c_void_p
    # 8193 drafter rows exceed the fixed scratch: rejected before anything is enqueued
    rc = lib.sdd_confidence_noalloc(VP(256), 1, 8193, 1, 1024, 1024, VP(256), VP(256), None, None, None, None, None,
                                    None, None)
    assert rc == 1
    assert b"8192" in lib.sdd_last_error()

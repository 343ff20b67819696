"""Failure detection of the bounded device waits: the streaming kernel's wait
for a tile copy is made to run out (the test hook keeps the first warp's first
copy from ever being issued, so nothing completes its barrier), with a short
poll limit.  The call must return, report SDD_DEV_TIMEOUT in its device status
word without trapping, and leave the context, the workspace and the next calls
correct (against the oracle)."""
import time

import numpy as np
import pytest
import torch

from paper_2608_14787_gb300 import synth
from parity_util import assert_close_stats

pytestmark = pytest.mark.gpu


def _check_against_oracle(orc, blk, conf):
    st = orc.row_stats(synth.bf16_bits(blk.z_d), tokens=blk.x.cpu().numpy())
    for name in ("q", "maxprob", "entropy"):
        assert_close_stats(name, getattr(conf, name), getattr(st, name), torch.bfloat16)
    np.testing.assert_array_equal(conf.argmax.cpu().numpy(), st.argmax)


@pytest.mark.parametrize("polls", [64, 4096])
def test_ring_wait_runs_out_and_recovers(sdd, orc, polls):
    blk = synth.make_block("c3", device="cuda", B=3, gamma=6, V=50_000)
    ws = sdd.Workspace(3, 6, 50_000)
    status = sdd.new_status()
    try:
        sdd.test_wait_hooks(polls, drop_copy=True)
        t0 = time.perf_counter()
        sdd.confidence(blk.z_d, blk.x, ws=ws, status=status)
        torch.cuda.synchronize()
        dt = time.perf_counter() - t0
    finally:
        sdd.test_wait_hooks(0, drop_copy=False)
    assert int(status.item()) & sdd.DEV_TIMEOUT, int(status.item())
    assert dt < 30.0
    # the status reader reports it as a return code and clears the word
    code, bits = sdd.status_from_device(status, clear=True)
    assert code == sdd.binding.SDD_ERR_DEVICE and bits & sdd.DEV_TIMEOUT
    assert int(status.item()) == 0 and sdd.status_from_device(status) == (0, 0)
    # the context, the workspace and the library stay usable
    conf = sdd.confidence(blk.z_d, blk.x, ws=ws, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    _check_against_oracle(orc, blk, conf)
    rnd = sdd.BlockRound(3, 6, 50_000, taus=(0.9,), K_min=2)
    rnd.set_inputs(blk.z_d, blk.z_t, blk.x, seed=1, round_=0)
    rnd.run()
    torch.cuda.synchronize()
    assert int(rnd.status.item()) == 0


def test_short_limit_without_a_dropped_copy_is_harmless(sdd, orc):
    """A short limit alone may or may not run out (each poll can suspend the
    warp until the copy lands): either the results are right and the status is
    clean, or the status reports the timeout."""
    blk = synth.make_block("c3", device="cuda", B=2, gamma=5, V=40_000)
    status = sdd.new_status()
    try:
        sdd.test_wait_hooks(2, drop_copy=False)
        conf = sdd.confidence(blk.z_d, blk.x, status=status)
        torch.cuda.synchronize()
    finally:
        sdd.test_wait_hooks(0, drop_copy=False)
    st = int(status.item())
    assert st in (0, sdd.DEV_TIMEOUT)
    assert sdd.status_from_device(status)[1] == st
    if st == 0:
        _check_against_oracle(orc, blk, conf)

"""Failure detection: every wait in the kernels is bounded.

A stuck wait must end as an EVISEL_ETIMEOUT status the host reads, with the
device still usable afterwards -- checked without faulting, trapping or
hanging the GPU: evisel_selftest_wait runs the kernels' bounded wait on a
barrier whose phase nothing completes (a flag that nothing sets), with a short
limit. The CPU test checks the argument validation.
"""
import time

import numpy as np
import pytest

from paper_2608_05780_gb300 import _binding as B
from paper_2608_05780_gb300 import workloads as wl
from paper_2608_05780_gb300.build import build

EVISEL_ETIMEOUT = -6


def test_selftest_rejects_bad_arguments():
    build()
    lib = B.load()
    import ctypes
    status = ctypes.c_int(7)
    assert lib.evisel_selftest_wait(0, 0, None, ctypes.byref(status)) == -1
    assert lib.evisel_selftest_wait(2_000_000, 0, None, ctypes.byref(status)) == -1
    assert lib.evisel_selftest_wait(1000, 0, None, None) == -1
    assert status.value == 7          # nothing ran


@pytest.mark.gpu
def test_stuck_wait_times_out_and_device_stays_usable(cuda_lib):
    import torch
    from gpu_helpers import check_o, run_cuda

    # A completed phase passes at once.
    assert B.evisel_selftest_wait(20_000, arrive=True) == 0
    # A phase nothing completes: the bounded wait gives up after ~20 ms.
    t0 = time.perf_counter()
    assert B.evisel_selftest_wait(20_000, arrive=False) == EVISEL_ETIMEOUT
    waited = time.perf_counter() - t0
    assert 0.015 < waited < 5.0, waited
    # The context is intact: a normal probe still matches the oracle.
    import oracle
    probe = wl.make_probe(wl.CONFIGS["tiny"])
    out, ws = run_cuda(cuda_lib, probe)
    assert B.evisel_status(ws) == 0
    o_ref, _ = oracle.probe(probe.q, probe.k, probe.v, probe.cu_seqlens, probe.n_vis, probe.cfg.tile,
                            probe.row_ptr, probe.col_idx)
    check_o(out["o"].float().cpu().numpy(), o_ref, "after a timed-out wait")
    ws.free()
    torch.cuda.synchronize()

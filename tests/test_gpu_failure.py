"""Failure detection on the GPU without a fault: a kernel's bounded wait on a
barrier that nothing signals gives up after its budget, the host reads
DAVET_ERR_TIMEOUT from the device error word, and the context keeps working
(the next call of the hot path runs and matches the oracle)."""
import numpy as np
import pytest
import torch

import oracle
from helpers import bits
from paper_2608_01821_gb300 import workloads

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_the_context_stays_usable(davet):
    davet.davet_device_status(clear=True)
    gave_up = torch.zeros(1, dtype=torch.int32, device="cuda")
    davet.davet_selftest_wait_timeout(gave_up)
    st, flags = davet.davet_device_status(clear=True)
    assert int(gave_up.item()) == 1
    assert st == 4 and flags & 0x1  # DAVET_ERR_TIMEOUT, the timeout bit
    assert davet.davet_device_status() == (0, 0)  # cleared
    # the context still runs the hot path: a pyramid build matches the oracle
    w = workloads.make("tiny")
    f = workloads.features(w, 0)
    side, off = davet.davet_pyramid_layout(w.grid, w.n_levels, 1)
    p = torch.empty((off[-1], w.C), dtype=torch.bfloat16, device="cuda")
    p[: off[1]].copy_(f.reshape(-1, w.C))
    davet.davet_build_pyramid(p, p, 1, w.grid, w.n_levels, w.C)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    ref = oracle.pyramid(f, 1, w.grid, w.n_levels, w.C)
    got = p.float().cpu().double().numpy()
    assert np.abs(got - ref).max() <= np.abs(ref).max() * 2.0 ** -7

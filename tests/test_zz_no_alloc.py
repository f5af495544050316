"""The allocation-free unmasking entry point (davet_unmask_topk_noalloc).

Some callers of this library cannot allocate device memory: a plugin that
only receives input and output buffers from an engine that owns all device
memory, or a serving loop that must not call cudaMalloc because it can
synchronize the device.  For them the library offers one entry point that
uses a fixed scratch array of its own instead of a caller workspace.

These tests call it through the C ABI and compare it with the workspace
entry point davet_unmask_topk on the same inputs, over two calls in a row
(the second call sees the scratch contents the first left behind), with the
same tolerances as the other unmasking tests.  The file sorts last so that a
run that stops at the first failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from helpers import TOPK_REL
from paper_2608_01821_gb300 import davet as davet_mod
from paper_2608_01821_gb300 import workloads

pytestmark = pytest.mark.gpu


def _state(resp, k, dev="cuda"):
    R = int(sum(resp))
    return dict(
        cu=torch.tensor(np.concatenate([[0], np.cumsum(resp)]), dtype=torch.int32, device=dev),
        masked=torch.ones(R, dtype=torch.uint8, device=dev),
        tokens=torch.full((R,), -1, dtype=torch.int32, device=dev),
        argmax=torch.full((R,), -1, dtype=torch.int32, device=dev),
        conf=torch.zeros(R, dtype=torch.float32, device=dev),
        committed=torch.zeros((len(resp), k), dtype=torch.int32, device=dev),
        stats=torch.zeros((len(resp), 2), dtype=torch.float32, device=dev),
    )


def _compare(a, b):
    assert torch.equal(a["argmax"], b["argmax"])
    assert torch.equal(a["masked"], b["masked"])
    assert torch.equal(a["tokens"], b["tokens"])
    assert torch.equal(a["committed"], b["committed"])
    ca, cb = a["conf"].double().cpu().numpy(), b["conf"].double().cpu().numpy()
    np.testing.assert_allclose(ca, cb, rtol=TOPK_REL, atol=0)
    np.testing.assert_allclose(a["stats"].cpu().numpy(), b["stats"].cpu().numpy(), rtol=TOPK_REL, atol=1e-7)


SCRATCH_BYTES = 1 << 20  # DAVET_NOALLOC_SCRATCH_BYTES


def _a256(n):
    return (n + 255) // 256 * 256


def _noalloc_max_rows():
    """Largest answer-row count the scratch array holds with one vocabulary
    chunk per row: 16-byte chunk records, 4-byte confidences and 4-byte
    indices, each array starting on a 256-byte boundary (the layout the
    header states)."""
    r = SCRATCH_BYTES // 24
    while _a256(16 * r) + 2 * _a256(4 * r) > SCRATCH_BYTES:
        r -= 1
    return r


def _logits(R, V, seed, dev):
    """Seeded N(0, 2) logits made on the device in row blocks (no fp32 copy
    of the whole matrix)."""
    out = torch.empty((R, V), dtype=torch.bfloat16, device=dev)
    g = torch.Generator(device=dev).manual_seed(seed)
    step = max(1, (1 << 28) // max(V, 1))
    for r0 in range(0, R, step):
        r1 = min(R, r0 + step)
        out[r0:r1] = (torch.randn((r1 - r0, V), generator=g, device=dev) * 1.4142135).to(torch.bfloat16)
    return out


@pytest.mark.parametrize("resp,V,k", [
    ([128], workloads.VOCAB_8B, 2),          # one 8B-class request (vocabulary split path)
    ([300, 0, 57, 512, 9], 4096, 3),         # ragged batch with an empty request
    ([32], 1024, 4),                         # tiny workload shape
    # the standard layout (16 chunks of 16 KB per row from 512 rows on) does
    # not fit: fewer, longer chunks
    ([5000], workloads.VOCAB_8B, 2),         # 12 chunks per row
    ([20000, 9000], workloads.VOCAB_8B, 2),  # one chunk per row; requests above the select's shared-memory rows
    ([_noalloc_max_rows()], 1024, 2),        # exactly the largest size the array holds
])
def test_noalloc_matches_workspace_entry_point_on_two_calls(davet, resp, V, k):
    dev = torch.device("cuda")
    R = int(sum(resp))
    B = len(resp)
    ref = _state(resp, k)
    new = _state(resp, k)
    ws_bytes = davet.davet_unmask_topk_workspace(R, V, B)
    if V == workloads.VOCAB_8B and R > 3970:
        # the workspace entry point's layout does not fit in the array, so the
        # allocation-free call runs on fewer vocabulary chunks per row
        assert ws_bytes > SCRATCH_BYTES
    ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device=dev)
    for call in range(2):
        lg = _logits(R, V, R + V + k + call, dev)
        davet.davet_unmask_topk(lg, V, ref["cu"], B, R, k, ref["masked"], ref["tokens"], ref["argmax"],
                                ref["conf"], ref["committed"], ref["stats"], ws)
        davet.davet_unmask_topk_noalloc(lg, V, new["cu"], B, R, k, new["masked"], new["tokens"], new["argmax"],
                                        new["conf"], new["committed"], new["stats"])
        torch.cuda.synchronize()
        assert davet.davet_device_status() == (0, 0)
        _compare(ref, new)
    # two commit rounds happened
    assert int((new["masked"] == 0).sum()) == sum(min(r, 2 * k) for r in resp)


def test_noalloc_rejects_sizes_beyond_its_scratch(davet):
    """One row more than the one-chunk layout holds (24 bytes per row) is
    rejected before anything is enqueued; the pointers are never read."""
    lib = davet_mod.load_cdll()
    p = torch.empty(16, dtype=torch.uint8, device="cuda")
    for too_many_rows, V in ((_noalloc_max_rows() + 1, 1024), (_noalloc_max_rows() + 1, workloads.VOCAB_8B),
                             (200000, workloads.VOCAB_8B)):
        n = ctypes.c_size_t(0)
        assert lib.davet_unmask_topk_workspace(too_many_rows, V, 1, ctypes.byref(n)) == 0
        assert n.value > SCRATCH_BYTES
        st = lib.davet_unmask_topk_noalloc(p.data_ptr(), V, p.data_ptr(), 1, too_many_rows, 2,
                                           p.data_ptr(), p.data_ptr(), None, None, None, None, None)
        assert st == davet_mod.ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)

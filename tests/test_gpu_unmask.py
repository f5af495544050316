"""Parity of davet_unmask_topk (Sec. 3.1, Eq. 1-2; Eq. 7 statistics) with
the fp64 oracle.

argmax is bit-exact (ties compare bf16 values exactly and resolve to the
lowest index on both sides); conf is within 1e-5 relative; the committed set
matches exactly unless the oracle's k-th and (k+1)-th confidences are within
1e-5 relative, in which case every pick must be within that margin of the
k-th; the answer state follows from the committed set; the mean confidence
and churn match within 1e-5.
"""
import numpy as np
import pytest
import torch

import oracle
from helpers import TOPK_REL, check_topk
from paper_2608_01821_gb300 import workloads

pytestmark = pytest.mark.gpu


class State:
    def __init__(self, resp, V, k, dev="cuda"):
        self.cu = np.concatenate([[0], np.cumsum(resp)]).astype(np.int32)
        R = int(self.cu[-1])
        self.R, self.V, self.k, self.B = R, V, k, len(resp)
        self.masked = np.ones(R, np.uint8)
        self.tokens = np.full(R, -1, np.int32)
        self.argmax = np.full(R, -1, np.int32)
        self.d = dict(
            cu=torch.from_numpy(self.cu).to(dev),
            masked=torch.ones(R, dtype=torch.uint8, device=dev),
            tokens=torch.full((R,), -1, dtype=torch.int32, device=dev),
            argmax=torch.full((R,), -1, dtype=torch.int32, device=dev),
            conf=torch.zeros(R, dtype=torch.float32, device=dev),
            committed=torch.zeros((self.B, k), dtype=torch.int32, device=dev),
            stats=torch.zeros((self.B, 2), dtype=torch.float32, device=dev),
        )

    def step(self, davet, logits_cpu):
        d = self.d
        ws = torch.zeros(max(davet.davet_unmask_topk_workspace(self.R, self.V, self.B), 256), dtype=torch.uint8,
                         device="cuda")
        davet.davet_unmask_topk(logits_cpu.cuda(), self.V, d["cu"], self.B, self.R, self.k, d["masked"],
                                d["tokens"], d["argmax"], d["conf"], d["committed"], d["stats"], ws)
        torch.cuda.synchronize()
        assert davet.davet_device_status() == (0, 0)
        prev_masked = self.masked.copy()
        conf_ref, com_ref, st_ref = oracle.unmask(logits_cpu, self.V, self.cu, self.k, self.masked, self.tokens,
                                                  self.argmax)
        m_rows = np.nonzero(prev_masked)[0]
        # argmax bit-exact, conf within 1e-5 relative
        g_arg = d["argmax"].cpu().numpy()
        assert np.array_equal(g_arg[m_rows], self.argmax[m_rows])
        g_conf = d["conf"].cpu().numpy().astype(np.float64)
        np.testing.assert_allclose(g_conf[m_rows], conf_ref[m_rows], rtol=TOPK_REL)
        # committed sets per request
        g_com = d["committed"].cpu().numpy()
        near = 0
        for b in range(self.B):
            rows_b = [i for i in m_rows if self.cu[b] <= i < self.cu[b + 1]]
            cref = {int(i - self.cu[b]): conf_ref[i] for i in rows_b}
            picks = [int(x) for x in g_com[b] if x >= 0]
            assert all(x == -1 for x in g_com[b][len(picks):])
            near += check_topk(picks, cref, self.k)
        # answer state follows the GPU commits (identical when no near tie)
        g_masked = d["masked"].cpu().numpy()
        g_tokens = d["tokens"].cpu().numpy()
        if not near:
            assert np.array_equal(g_masked, self.masked)
            assert np.array_equal(g_tokens, self.tokens)
        else:
            # in a near tie the oracle's state follows the GPU's valid choice
            self.masked[:] = g_masked
            self.tokens[:] = g_tokens
        np.testing.assert_allclose(d["stats"].cpu().numpy(), st_ref, rtol=TOPK_REL, atol=1e-7)
        return near


def test_tiny_workload_all_steps(davet):
    w = workloads.make("tiny")
    s = State(w.resp, w.V, w.k)
    for t in range(w.T):
        s.step(davet, workloads.logits(w, t))
    assert s.masked.sum() == 0  # 32 rows, 4 per step, 8 steps


def test_single_workload_first_steps(davet):
    w = workloads.make("single")
    s = State(w.resp, w.V, w.k)
    for t in range(3):
        s.step(davet, workloads.logits(w, t))


def test_ragged_requests_with_fewer_than_k_left(davet):
    resp = [3, 0, 17, 1, 40]
    V, k = 2048, 4
    s = State(resp, V, k)
    g = torch.Generator().manual_seed(3)
    for t in range(6):
        lg = (torch.randn((sum(resp), V), generator=g) * 1.4142).to(torch.bfloat16)
        s.step(davet, lg)


def test_ties_resolve_to_lowest_index_and_position(davet):
    V, k = 1024, 3
    resp = [8]
    lg = torch.zeros((8, V), dtype=torch.bfloat16)
    lg[:, 5] = 2.0
    lg[:, 700] = 2.0       # tied max: argmax must be 5
    lg[3, 9] = 2.0         # row 3 has a lower-probability max (three tied)
    s = State(resp, V, k)
    s.step(davet, lg)
    com = s.d["committed"].cpu().numpy()[0]
    # rows 0,1,2,4.. have equal conf: lowest positions first, row 3 is lower
    assert list(com) == [0, 1, 2]
    assert (s.d["argmax"].cpu().numpy() == 5).all()


def test_argmax_ties_inside_one_lane_batch(davet):
    """Equal maxima planted where the row pass must order them itself.

    At V = 126464 and 8 rows a row has 31 vocabulary chunks of 510 16-byte
    slices; a lane folds its 8 slices of a 256-slice piece (slices
    lane + 32 m) as one batch when all 8 exist, else slice by slice.  The
    maxima sit in two slices of one batch, twice in one slice, in two lanes,
    in two chunks, in a partial piece after a full one, and as a later,
    larger maximum (the rescale).  argmax must be the first index of the
    maximum (Eq. 1 reads the arg-max token; ties take the lowest index, as in
    the oracle), conf as in the oracle.  Should the chunking change, the
    comparison with the oracle still holds."""
    V, k, chunk = 126464, 2, 510

    def el(ch, piece, lane, m, pos):
        return (ch * chunk + piece * 256 + lane + 32 * m) * 8 + pos

    plants = {
        0: [(el(0, 0, 3, 5, 1), 8.0), (el(0, 0, 3, 2, 5), 8.0)],     # two slices of one batch
        1: [(el(2, 0, 9, 4, 6), 8.0), (el(2, 0, 9, 4, 2), 8.0)],     # one slice, two positions
        2: [(el(5, 0, 7, 0, 3), 8.0), (el(5, 0, 2, 1, 0), 8.0)],     # two lanes of one piece
        3: [(el(3, 0, 0, 0, 0), 8.0), (el(1, 1, 4, 3, 7), 8.0)],     # two chunks
        4: [(el(4, 1, 31, 6, 4), 8.0), (el(4, 0, 30, 7, 1), 8.0)],   # partial piece after a full one
        5: [(el(6, 0, 5, 1, 1), 6.0), (el(6, 1, 5, 1, 1), 8.0)],     # a later, larger maximum
        6: [(el(30, 1, 10, 6, 0), 8.0)],                              # the last chunk
        7: [],
    }
    g = torch.Generator().manual_seed(11)
    lg = torch.randn((8, V), generator=g) * 0.5
    expect = {}
    for r, pl in plants.items():
        for pos, val in pl:
            assert 0 <= pos < V
            lg[r, pos] = val
        if pl:
            top = max(v for _, v in pl)
            expect[r] = min(p for p, v in pl if v == top)
    lg = lg.to(torch.bfloat16)
    s = State([8], V, k)
    s.step(davet, lg)
    arg = s.d["argmax"].cpu().numpy()
    for r, e in expect.items():
        assert arg[r] == e, (r, int(arg[r]), e)


def test_churn_and_mean_confidence(davet):
    V, k = 64, 1
    resp = [4]
    s = State(resp, V, k)
    lg0 = torch.zeros((4, V), dtype=torch.bfloat16)
    for i in range(4):
        lg0[i, i] = 3.0
    s.step(davet, lg0)  # first step: churn 0
    assert s.d["stats"].cpu().numpy()[0, 1] == 0.0
    lg1 = lg0.clone()
    lg1[1, 1] = 0.0
    lg1[1, 40] = 3.0    # row 1 changes its argmax
    s.step(davet, lg1)
    # row 0 was committed at step 0 (ties -> lowest position); rows 1..3
    # remain, all had a previous prediction, one changed
    assert abs(s.d["stats"].cpu().numpy()[0, 1] - 1 / 3) < 1e-7


@pytest.mark.parametrize("name", ["highres", "ragged"])
def test_full_size_first_step(davet, name):
    w = workloads.make(name)
    s = State(w.resp, w.V, w.k)
    s.step(davet, workloads.logits(w, 0))


def test_host_mapped_logits_match_device_logits(davet):
    """Logits in pinned host memory (read by the kernels over the host link,
    masked rows only) give bit-identical results to the same logits in device
    memory, over three steps of an 8B-class vocabulary."""
    resp, V, k = [40, 7, 81], workloads.VOCAB_8B, 3
    a, b = State(resp, V, k), State(resp, V, k)
    for t in range(3):
        lg = workloads.normal_bf16((a.R, V), 900 + t, 2 ** 0.5)
        host = lg.pin_memory()
        for st, src in ((a, lg.cuda()), (b, host)):
            d = st.d
            ws = torch.zeros(max(davet.davet_unmask_topk_workspace(st.R, V, st.B), 256), dtype=torch.uint8,
                             device="cuda")
            davet.davet_unmask_topk(src, V, d["cu"], st.B, st.R, k, d["masked"], d["tokens"], d["argmax"],
                                    d["conf"], d["committed"], d["stats"], ws)
        torch.cuda.synchronize()
        assert davet.davet_device_status() == (0, 0)
        for key in ("masked", "tokens", "argmax", "conf", "committed", "stats"):
            assert torch.equal(a.d[key], b.d[key]), (t, key)


@pytest.mark.parametrize("V,src_host", [(workloads.VOCAB_8B, True), (workloads.VOCAB_8B, False), (1024, True),
                                        (4104, False)])
def test_stage_masked_rows_copies_exactly_the_masked_rows(davet, V, src_host):
    """davet_stage_masked_rows: every masked row bit for bit (from pinned host
    or device memory, a vocabulary that is not a multiple of the chunk), every
    other row of the destination untouched, nothing for an all-clear mask."""
    R = 37
    lg = workloads.normal_bf16((R, V), 950 + V, 2 ** 0.5)
    src = lg.pin_memory() if src_host else lg.cuda()
    g = torch.Generator().manual_seed(V)
    masked = (torch.rand(R, generator=g) < 0.6).to(torch.uint8)
    masked[0], masked[-1] = 1, 0
    dst = torch.full((R, V), -3.0, dtype=torch.bfloat16, device="cuda")
    davet.davet_stage_masked_rows(src, V, masked.cuda(), R, dst)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    m = masked.bool()
    out = dst.cpu()
    assert torch.equal(out[m].view(torch.int16), lg[m].view(torch.int16))
    assert (out[~m].float() == -3.0).all()
    davet.davet_stage_masked_rows(src, V, torch.zeros(R, dtype=torch.uint8, device="cuda"), R, dst)
    torch.cuda.synchronize()
    assert torch.equal(dst.cpu().view(torch.int16), out.view(torch.int16))

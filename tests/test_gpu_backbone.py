"""The full backbone step (paper_2608_01821_gb300/model.py) against the fp64
layer oracle: step inputs [view || prompt || answer embeddings], n layers,
final normalization and LM head; then a closed denoising loop."""
import numpy as np
import pytest
import torch

import oracle
from oracle import layer as L
from paper_2608_01821_gb300 import workloads
from paper_2608_01821_gb300.model import RMS_EPS, ROPE_THETA, Backbone

pytestmark = pytest.mark.gpu


def f64(t):
    return t.detach().cpu().double().numpy()


def oracle_inputs(bb, feats, prompts, t):
    """Packed step input as the oracle builds it: the step's pooled view
    (fp64 means rounded to bf16), the prompt rows, the mask embedding."""
    w = bb.w
    C = bb.C
    rows, cu = [], [0]
    sides = w.level_sides()
    for b in range(w.batch):
        lvl = int(w.schedule[t, b])
        parts = []
        if w.tiles[b]:
            pyr = torch.from_numpy(oracle.pyramid(feats[b], w.tiles[b], w.grid, w.n_levels, C)).to(torch.bfloat16)
            if lvl < w.n_levels:
                off = oracle.level_offsets(w.grid, w.n_levels, w.tiles[b])
                view = pyr[off[lvl]:off[lvl + 1]]
            else:  # the mixed view, from the oracle's own bf16 pyramid
                bits = oracle.mixed_view(pyr.view(torch.int16).numpy().view(np.uint16), w.tiles[b], w.grid,
                                         w.n_levels, *w.mixed, C)
                view = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16)
            parts.append(f64(view))
        parts.append(f64(prompts[b]))
        parts.append(np.repeat(f64(bb.emb[bb.mask_id:bb.mask_id + 1]), w.resp[b], axis=0))
        x = np.concatenate(parts)
        rows.append(x)
        cu.append(cu[-1] + len(x))
    return np.concatenate(rows), cu


def layer_weights(p, F):
    """The oracle's layer weights from the model's: the normalization gains
    are folded into the QKV and gate/up weights the model holds
    (rmsnorm(x, g) W^T = rmsnorm(x, 1) (W diag g)^T), so the oracle takes
    those bf16 weights with unit gains."""
    C = p["g1"].numel()
    wqkv = f64(p["wqkv"])
    HD = wqkv.shape[0] // 3
    gu = f64(p["wgu"]).reshape(F // 128, 2, 128, C)
    return dict(g1=np.ones(C), wq=wqkv[:HD], wk=wqkv[HD:2 * HD], wv=wqkv[2 * HD:], wo=f64(p["wo"]), g2=np.ones(C),
                wg=gu[:, 0].reshape(F, C), wu=gu[:, 1].reshape(F, C), wd=f64(p["wd"]))


@pytest.mark.parametrize("name,t,device_rows", [("tiny", 0, False), ("tiny", 2, False), ("tiny", 5, False),
                                                ("tiny", 2, True), ("tiny", 5, True), ("tiny_mixed", 2, False),
                                                ("tiny_mixed", 3, True)])
def test_tiny_two_layer_step_logits(davet, name, t, device_rows):
    """device_rows: the policy's launch mode, every kernel launched for the
    largest view and reading the step's row count on the device (the step's
    view still comes from the workload's schedule here).  tiny_mixed steps 2
    and 3 take the mixed view (coarse rows plus the level-0 lattice)."""
    w = workloads.make(name)
    bb = Backbone(w, 2, lib=davet)
    if device_rows:
        bb.use_policy()
        assert bb.rows(t) < bb.max_rows
    feats = [workloads.normal_bf16((w.tiles[b], w.grid, w.grid, bb.C), 100 + b) for b in range(w.batch)]
    prompts = [workloads.normal_bf16((w.prompt[b], bb.C), 200 + b) for b in range(w.batch)]
    bb.load_inputs(feats, prompts)
    bb.reset_state()
    bb.build_pyramids()
    bb.forward(t)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    x, cu = oracle_inputs(bb, feats, prompts, t)
    assert list(bb.cu.cpu().numpy()) == cu
    for p in bb.layers:
        x = L.layer(x, layer_weights(p, bb.F), cu, w.H, w.D, ROPE_THETA, RMS_EPS)
    ref = L.answer_logits(x, cu, w.resp, f64(bb.gf), f64(bb.wlm), RMS_EPS)
    got = f64(bb.logits[: bb.R])
    rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
    assert rel < 3e-2, rel
    # the committed choice follows the logits: argmax agreement on rows with a clear margin
    top2 = np.sort(ref, axis=1)[:, -2:]
    clear = (top2[:, 1] - top2[:, 0]) > 0.05 * np.abs(top2[:, 1])
    assert (got.argmax(1)[clear] == ref.argmax(1)[clear]).all()


def test_closed_loop_commits_every_position(davet):
    """T steps of k commits: every answer position ends committed, each step
    commits only still-masked positions, and every token is a vocabulary id
    (the mask id never wins a commit only by chance, so it is not excluded)."""
    w = workloads.make("tiny")
    bb = Backbone(w, 1, lib=davet)
    feats = [workloads.normal_bf16((w.tiles[b], w.grid, w.grid, bb.C), 300 + b) for b in range(w.batch)]
    prompts = [workloads.normal_bf16((w.prompt[b], bb.C), 400 + b) for b in range(w.batch)]
    bb.load_inputs(feats, prompts)
    bb.reset_state()
    bb.build_pyramids()
    for t in range(w.T):
        bb.step(t)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    committed = bb.committed.cpu().numpy()
    assert (committed >= 0).all()
    flat = committed.reshape(-1)
    assert len(set(flat.tolist())) == len(flat) == w.T * w.k  # every position once
    assert int(bb.masked.sum()) == w.total_resp - w.T * w.k
    tok = bb.tokens.cpu().numpy()
    assert ((tok[flat] >= 0) & (tok[flat] < w.V)).all()


@pytest.mark.parametrize("orientation,B,rho,alpha,uniform", [("early", 0.75, 0.2, 1.0, False),
                                                             ("late", 0.45, 0.2, 0.5, True)])
def test_policy_closed_loop(davet, orientation, B, rho, alpha, uniform):
    """The allocation policy picks every step's view on the device from the
    previous step's statistics; the steps run the rows of the views it picked
    (cu_seqlens of the last step) and the loop commits every position.  The
    budgets stay inside the envelope's bounds (Eq. 8 interpolates them)."""
    w = workloads.make("tiny")
    bb = Backbone(w, 1, lib=davet)
    bb.use_policy(orientation, B, rho, alpha, uniform_demand=uniform)
    feats = [workloads.normal_bf16((w.tiles[b], w.grid, w.grid, bb.C), 500 + b) for b in range(w.batch)]
    prompts = [workloads.normal_bf16((w.prompt[b], bb.C), 600 + b) for b in range(w.batch)]
    bb.load_inputs(feats, prompts)
    bb.begin_pass()
    bb.build_pyramids()
    for t in range(w.T):
        bb.step(t)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    sched = bb.schedule.cpu().numpy()
    assert set(np.unique(sched).tolist()) <= set(workloads.policy_view_levels(w))
    cu = bb.cu.cpu().numpy()
    assert int(cu[-1]) == bb.rows_of(sched[-1])
    assert [int(cu[b + 1] - cu[b]) for b in range(w.batch)] == [w.seq_len(b, int(v)) for b, v in enumerate(sched[-1])]
    committed = bb.committed.cpu().numpy().reshape(-1)
    assert len(set(committed.tolist())) == len(committed) == w.T * w.k
    budget = bb.budget.cpu().numpy()  # [T][batch]
    lo, up = bb.lo.cpu().numpy().T, bb.up.cpu().numpy().T  # [T][batch]
    assert ((budget >= lo - 1e-12) & (budget <= up + 1e-12)).all()
    assert ((budget >= 0) & (budget <= 1)).all()

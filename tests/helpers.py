"""Shared test utilities: bf16 views, the tolerance checks of the parity
tests, and the top-k near-tie rule."""
import numpy as np
import torch

# attention tolerances for bf16 inputs (fp32 accumulation, bf16 output)
ATTN_MAX_ABS = 1e-2
ATTN_REL_L2 = 5e-3
# pooled values: relative to the window's mean |x|
POOL_REL = 1e-6
# confidence near-tie margin for the top-k comparison (fp32 vs fp64)
TOPK_REL = 1e-5


def bits(t: torch.Tensor) -> np.ndarray:
    """uint16 bit patterns of a bf16 tensor (CPU copy)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def bf16_to_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().float().double().numpy()


def check_bf16_rounding(gpu_bf16: np.ndarray, ref: np.ndarray, scale: np.ndarray, tol=POOL_REL):
    """gpu must be RNE(ref), or a neighbour when ref lies within tol*scale of
    the rounding midpoint: |gpu - ref| <= ulp(ref)/2 + tol*scale."""
    a = np.abs(ref)
    e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    ulp = np.where(a > 0, 2.0 ** (e - 7), 2.0 ** -133)
    bad = np.abs(gpu_bf16 - ref) > 0.5 * ulp + tol * scale + 1e-300
    return int(bad.sum())


def attn_errors(gpu: np.ndarray, ref: np.ndarray):
    d = gpu - ref
    max_abs = float(np.abs(d).max()) if d.size else 0.0
    rel_l2 = float(np.linalg.norm(d) / max(np.linalg.norm(ref), 1e-30)) if d.size else 0.0
    return max_abs, rel_l2


def check_topk(gpu_set, conf_ref: dict, k: int):
    """Compare the committed set of one request against fp64 confidences.

    conf_ref maps row -> oracle conf for the rows of M_t.  Exact set equality
    is required when the oracle's gap between ranks k and k+1 exceeds
    TOPK_REL relative; otherwise every pick must lie within TOPK_REL of the
    k-th oracle confidence.  Returns True when the near-tie rule was used."""
    order = sorted(conf_ref, key=lambda i: (-conf_ref[i], i))
    take = min(k, len(order))
    want = set(order[:take])
    assert len(gpu_set) == take
    if take == len(order):
        assert set(gpu_set) == want
        return False
    ck, ck1 = conf_ref[order[take - 1]], conf_ref[order[take]]
    if ck - ck1 > TOPK_REL * ck:
        assert set(gpu_set) == want, (sorted(gpu_set), sorted(want))
        return False
    for i in gpu_set:
        assert conf_ref[i] >= ck - TOPK_REL * ck
    return True

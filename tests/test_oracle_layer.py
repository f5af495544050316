"""Pins for the full-layer oracle (oracle/layer.py): library functions for
the normalization and the activation, identities of the rotary embedding,
and closed forms of the layer in special cases."""
import numpy as np
import pytest
import torch

from oracle import layer as L


def test_rmsnorm_matches_torch_and_closed_form():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((7, 48))
    g = rng.standard_normal(48)
    ref = torch.nn.functional.rms_norm(torch.from_numpy(x), (48,), torch.from_numpy(g), eps=1e-5).numpy()
    assert np.allclose(L.rmsnorm(x, g, 1e-5), ref, rtol=1e-12, atol=1e-12)
    # a constant row c normalizes to sign(c) * |c| / sqrt(c^2 + eps) * gamma
    c = np.full((1, 16), -3.0)
    assert np.allclose(L.rmsnorm(c, np.ones(16), 1e-5), -3.0 / np.sqrt(9.0 + 1e-5))
    # scale invariance (eps = 0)
    assert np.allclose(L.rmsnorm(5.0 * x, g, 0.0), L.rmsnorm(x, g, 0.0))


def test_silu_matches_torch():
    g = np.linspace(-30, 30, 601)
    assert np.allclose(L.silu(g), torch.nn.functional.silu(torch.from_numpy(g)).numpy(), rtol=1e-12, atol=1e-15)
    assert L.silu(np.array([0.0]))[0] == 0.0


@pytest.mark.parametrize("D", [64, 128])
def test_rope_identities(D):
    rng = np.random.default_rng(D)
    H, n = 3, 9
    x = rng.standard_normal((n, H * D))
    pos = np.arange(n) * 37
    y = L.rope(x, pos, H, D, 500000.0)
    # position 0 is the identity
    assert np.allclose(L.rope(x[:1], [0], H, D, 500000.0), x[:1])
    # every rotated pair keeps its length
    half = D // 2
    xh, yh = x.reshape(n, H, D), y.reshape(n, H, D)
    assert np.allclose(xh[..., :half] ** 2 + xh[..., half:] ** 2, yh[..., :half] ** 2 + yh[..., half:] ** 2)
    # the first pair turns by exactly the position (theta^0 = 1), as a complex product
    z = (xh[..., 0] + 1j * xh[..., half]) * np.exp(1j * pos)[:, None]
    assert np.allclose(yh[..., 0], z.real) and np.allclose(yh[..., half], z.imag)
    # dot products depend only on the position difference
    q, k = rng.standard_normal((1, H * D)), rng.standard_normal((1, H * D))
    d1 = (L.rope(q, [5], H, D, 1e4) * L.rope(k, [2], H, D, 1e4)).sum()
    d2 = (L.rope(q, [105], H, D, 1e4) * L.rope(k, [102], H, D, 1e4)).sum()
    assert np.isclose(d1, d2)


def weights(rng, C, HD, F, zero=()):
    w = dict(g1=1 + 0.1 * rng.standard_normal(C), wq=rng.standard_normal((HD, C)) / np.sqrt(C),
             wk=rng.standard_normal((HD, C)) / np.sqrt(C), wv=rng.standard_normal((HD, C)) / np.sqrt(C),
             wo=rng.standard_normal((C, HD)) / np.sqrt(HD), g2=1 + 0.1 * rng.standard_normal(C),
             wg=rng.standard_normal((F, C)) / np.sqrt(C), wu=rng.standard_normal((F, C)) / np.sqrt(C),
             wd=rng.standard_normal((C, F)) / np.sqrt(F))
    for k in zero:
        w[k] = np.zeros_like(w[k])
    return w


def test_zero_output_projections_give_the_identity():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((10, 32))
    w = weights(rng, 32, 32, 64, zero=("wo", "wd"))
    assert np.array_equal(L.layer(x, w, [0, 4, 10], 4, 8, 1e4, 1e-5), x)


def test_equal_scores_average_each_request_separately():
    """With zero query and key weights every score is 0, so each row's
    attention output is the mean value of its own request (no causal mask,
    no mixing across requests)."""
    rng = np.random.default_rng(2)
    C, H, D = 32, 4, 8
    x = rng.standard_normal((9, C))
    w = weights(rng, C, H * D, 64, zero=("wq", "wk", "wd"))
    cu = [0, 3, 3, 9]
    got = L.layer(x, w, cu, H, D, 1e4, 1e-5)
    h = L.rmsnorm(x, w["g1"], 1e-5)
    v = h @ w["wv"].T
    want = x.copy()
    for b in range(3):
        s0, s1 = cu[b], cu[b + 1]
        if s1 > s0:
            want[s0:s1] += v[s0:s1].mean(axis=0) @ w["wo"].T
    assert np.allclose(got, want, rtol=1e-12, atol=1e-12)


def test_single_row_request_attends_to_itself_and_mlp_closed_form():
    rng = np.random.default_rng(3)
    C, H, D, F = 16, 2, 8, 32
    x = rng.standard_normal((1, C))
    w = weights(rng, C, H * D, F)
    got = L.layer(x, w, [0, 1], H, D, 1e4, 1e-5)
    h = L.rmsnorm(x, w["g1"], 1e-5)
    x1 = x + (h @ w["wv"].T) @ w["wo"].T  # one key: softmax weight 1 on itself
    h2 = L.rmsnorm(x1, w["g2"], 1e-5)
    g, u = h2 @ w["wg"].T, h2 @ w["wu"].T
    want = x1 + (g / (1 + np.exp(-g)) * u) @ w["wd"].T
    assert np.allclose(got, want, rtol=1e-12, atol=1e-12)


def test_answer_logits_take_the_last_rows_of_each_request():
    rng = np.random.default_rng(4)
    x = rng.standard_normal((12, 16))
    g = np.ones(16)
    w = rng.standard_normal((5, 16))
    out = L.answer_logits(x, [0, 5, 12], [2, 3], g, w, 0.0)
    rows = [3, 4, 9, 10, 11]
    assert np.allclose(out, L.rmsnorm(x[rows], g, 0.0) @ w.T)

"""Pins for the oracle's bidirectional step attention (Sec. 3.1, Eq. 1).

Closed forms and invariants that any correct softmax(scale * Q K^T) V over a
request's rows must satisfy: identical keys give the mean of the values, one
row gives its own value, two keys give a logistic mix, a dominant key selects
its value, and permuting a request's rows permutes its outputs.  Requests are
independent (no attention across the packed boundary), and there is no
causal mask.
"""
import math

import numpy as np
import pytest
import torch

import oracle


def bf(x):
    return torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)


def widen(t):
    return t.float().double().numpy()


def rand_qkv(n, H, D, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randn(n, 3, H, D, generator=g).to(torch.bfloat16)


def test_identical_keys_give_mean_of_values():
    H, D, L = 3, 16, 37
    qkv = rand_qkv(L, H, D, 1)
    qkv[:, 1] = qkv[0:1, 1]  # every key row equal
    cu = np.array([0, L], dtype=np.int32)
    out = oracle.attention(qkv, cu, H, D, 1 / math.sqrt(D))
    v = widen(qkv[:, 2])
    np.testing.assert_allclose(out, np.broadcast_to(v.mean(axis=0), out.shape), rtol=1e-12, atol=1e-13)


def test_single_row_returns_its_value():
    H, D = 2, 8
    qkv = rand_qkv(5, H, D, 2)
    cu = np.arange(6, dtype=np.int32)  # five requests of one row each
    out = oracle.attention(qkv, cu, H, D, 0.3)
    np.testing.assert_array_equal(out, widen(qkv[:, 2]))


def test_two_keys_logistic_closed_form():
    H, D = 1, 4
    q = [0.5, -1.0, 2.0, 0.25]
    k1 = [1.0, 0.5, -0.75, 2.0]
    k2 = [-0.5, 1.5, 0.125, 1.0]
    qkv = torch.zeros(2, 3, H, D, dtype=torch.bfloat16)
    qkv[0, 0, 0] = bf(q)
    qkv[1, 0, 0] = bf(k2)  # query of row 1 (arbitrary)
    qkv[0, 1, 0] = bf(k1)
    qkv[1, 1, 0] = bf(k2)
    qkv[0, 2, 0] = bf([1, 2, 3, 4])
    qkv[1, 2, 0] = bf([-4, 0.5, 8, -1])
    scale = 0.5
    out = oracle.attention(qkv, np.array([0, 2], np.int32), H, D, scale)
    s1 = scale * float(np.dot(q, k1))
    s2 = scale * float(np.dot(q, k2))
    w1 = 1.0 / (1.0 + math.exp(s2 - s1))
    expect = w1 * np.array([1, 2, 3, 4.0]) + (1 - w1) * np.array([-4, 0.5, 8, -1.0])
    np.testing.assert_allclose(out[0, 0], expect, rtol=1e-14, atol=1e-14)


def test_dominant_key_selects_its_value():
    H, D, L = 2, 8, 20
    qkv = rand_qkv(L, H, D, 3)
    qkv[:, 1] *= 0.01
    j = 13
    # every query along the all-ones direction; key j far along it
    qkv[:, 0] = bf(np.ones((L, H, D)))
    qkv[j, 1] = bf(np.full((H, D), 8.0))
    out = oracle.attention(qkv, np.array([0, L], np.int32), H, D, 1.0)
    v = widen(qkv[:, 2])
    np.testing.assert_allclose(out, np.broadcast_to(v[j], out.shape), rtol=0, atol=1e-12)


def test_permutation_equivariance():
    H, D, L = 2, 16, 29
    qkv = rand_qkv(L, H, D, 4)
    perm = np.random.default_rng(0).permutation(L)
    cu = np.array([0, L], np.int32)
    a = oracle.attention(qkv, cu, H, D, 0.25)
    b = oracle.attention(qkv[torch.as_tensor(perm)].contiguous(), cu, H, D, 0.25)
    np.testing.assert_allclose(b, a[perm], rtol=1e-12, atol=1e-13)


def test_requests_are_independent_and_non_causal():
    H, D = 2, 8
    qkv = rand_qkv(30, H, D, 5)
    cu = np.array([0, 12, 30], np.int32)
    both = oracle.attention(qkv, cu, H, D, 0.35)
    first = oracle.attention(qkv[:12].contiguous(), np.array([0, 12], np.int32), H, D, 0.35)
    second = oracle.attention(qkv[12:].contiguous(), np.array([0, 18], np.int32), H, D, 0.35)
    np.testing.assert_array_equal(both[:12], first)
    np.testing.assert_array_equal(both[12:], second)
    # non-causal: changing the last key changes the first row's output
    qkv2 = qkv.clone()
    qkv2[11, 1] = -qkv2[11, 1]
    changed = oracle.attention(qkv2, cu, H, D, 0.35)
    assert np.abs(changed[0] - both[0]).max() > 1e-6


def test_rows_variant_matches_dense():
    H, D = 4, 16
    qkv = rand_qkv(50, H, D, 6)
    cu = np.array([0, 7, 7, 50], np.int32)  # includes an empty request
    dense = oracle.attention(qkv, cu, H, D, 0.25)
    rows = np.array([0, 6, 7, 33, 49])
    heads = np.array([0, 3, 1, 2, 3])
    sampled = oracle.attention_rows(qkv, cu, H, D, 0.25, rows, heads)
    np.testing.assert_array_equal(sampled, dense[rows, heads])


def test_matches_library_softmax_on_random_input():
    # scipy's softmax and numpy matmul as the stepping stones
    sp = pytest.importorskip("scipy.special")
    H, D, L = 2, 32, 41
    qkv = rand_qkv(L, H, D, 8)
    x = widen(qkv)
    out = oracle.attention(qkv, np.array([0, L], np.int32), H, D, 0.2)
    for h in range(H):
        p = sp.softmax(0.2 * x[:, 0, h] @ x[:, 1, h].T, axis=1)
        np.testing.assert_allclose(out[:, h], p @ x[:, 2, h], rtol=1e-11, atol=1e-12)

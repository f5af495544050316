"""Pins for the oracle's confidence-ranked unmasking (Sec. 3.1, Eq. 1-2) and
its step statistics (Sec. 4.2, Eq. 7 inputs).

Closed-form confidences, the lowest-index argmax rule, a brute-force
enumeration of the top-k set, the "commit all when fewer than k remain"
case, and hand-counted churn.
"""
import itertools
import math

import numpy as np
import torch

import oracle


def bf_bits(x):
    t = torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def state(rows):
    return (np.ones(rows, np.uint8), np.full(rows, -7, np.int32), np.full(rows, -1, np.int32))


def test_uniform_row_conf_is_one_over_v_and_argmax_lowest():
    V = 1000
    lg = bf_bits(np.full((1, V), 0.5))
    m, tok, am = state(1)
    conf, com, st = oracle.unmask(lg, V, [0, 1], 1, m, tok, am)
    assert am[0] == 0 and tok[0] == 0 and m[0] == 0
    assert abs(conf[0] - 1.0 / V) < 1e-15
    assert com[0, 0] == 0
    assert abs(st[0, 0] - 1.0 / V) < 1e-15 and st[0, 1] == 0.0


def test_one_peak_closed_form():
    V, a, b, j = 4096, 3.0, -1.25, 777
    row = np.full(V, b)
    row[j] = a
    m, tok, am = state(1)
    conf, _, _ = oracle.unmask(bf_bits(row[None]), V, [0, 1], 1, m, tok, am)
    assert am[0] == j
    # sequential fp64 sum of V terms: relative error below V * 2^-53
    np.testing.assert_allclose(conf[0], 1.0 / (1.0 + (V - 1) * math.exp(b - a)), rtol=V * 2.0**-53)


def test_tied_max_takes_lowest_index():
    V = 64
    row = np.linspace(-2, 1, V)
    row[[5, 40, 63]] = 2.0
    m, tok, am = state(1)
    conf, _, _ = oracle.unmask(bf_bits(row[None]), V, [0, 1], 1, m, tok, am)
    assert am[0] == 5
    w = np.exp(torch.as_tensor(row, dtype=torch.float32).to(torch.bfloat16).double().numpy() - 2.0)
    np.testing.assert_allclose(conf[0], 1.0 / w.sum(), rtol=1e-14)


def test_softmax_row_sums_to_one_and_conf_is_max_prob():
    g = torch.Generator().manual_seed(1)
    V = 126464
    row = (torch.randn(V, generator=g) * math.sqrt(2)).to(torch.bfloat16)
    p = oracle.softmax_row(row)
    assert abs(p.sum() - 1.0) < 1e-12
    m, tok, am = state(1)
    conf, _, _ = oracle.unmask(row.view(1, V), V, [0, 1], 1, m, tok, am)
    assert conf[0] == p.max()
    assert 1.0 / V < conf[0] <= 1.0
    assert am[0] == int(np.argmax(p))


def _logits_with_confs(peaks, V=32):
    """Rows whose max softmax probability grows with `peaks` (one peak per row)."""
    rows = np.zeros((len(peaks), V))
    for i, a in enumerate(peaks):
        rows[i, i % V] = a
    return rows


def test_topk_brute_force_small():
    rng = np.random.default_rng(5)
    V = 32
    for trial in range(40):
        n = int(rng.integers(1, 11))
        k = int(rng.integers(1, 6))
        # peaks on a coarse grid so that ties occur and exercise the position rule
        peaks = rng.integers(0, 5, size=n) * 0.5
        lg = bf_bits(_logits_with_confs(peaks, V))
        masked = (rng.random(n) < 0.8).astype(np.uint8)
        m, tok, am = masked.copy(), np.full(n, -7, np.int32), np.full(n, -1, np.int32)
        conf, com, _ = oracle.unmask(lg, V, [0, n], k, m, tok, am)
        cand = [i for i in range(n) if masked[i]]
        take = min(k, len(cand))
        # the committed set is the unique subset that dominates every other
        # candidate under (higher conf, then lower position)
        key = {i: (conf[i], -i) for i in cand}
        winners = [set(s) for s in itertools.combinations(cand, take)
                   if all(key[a] > key[b] for a in s for b in cand if b not in s)]
        assert len(winners) == 1
        got = [c for c in com[0] if c >= 0]
        assert set(got) == winners[0]
        assert len(got) == take and all(c == -1 for c in com[0][take:])
        # rank order
        assert [key[i] for i in got] == sorted([key[i] for i in got], reverse=True)
        for i in range(n):
            if i in winners[0]:
                assert m[i] == 0 and tok[i] == am[i]
            else:
                assert m[i] == masked[i] and tok[i] == -7


def test_fewer_than_k_masked_commits_all_and_empty_request():
    V = 16
    rows = _logits_with_confs([1.0, 2.0, 0.5, 3.0, 1.5], V)
    masked = np.array([0, 1, 0, 1, 0], np.uint8)
    m, tok, am = masked.copy(), np.full(5, -7, np.int32), np.full(5, -1, np.int32)
    conf, com, st = oracle.unmask(bf_bits(rows), V, [0, 0, 5], 4, m, tok, am)
    assert (com[0] == -1).all() and st[0, 0] == 0 and st[0, 1] == 0  # empty request
    assert list(com[1]) == [3, 1, -1, -1]
    assert (m == 0).all()
    assert tok[1] == 1 and tok[3] == 3
    np.testing.assert_allclose(st[1, 0], (conf[1] + conf[3]) / 2, rtol=1e-15)


def test_churn_counts_rows_with_a_previous_prediction():
    V = 16
    rows = np.zeros((6, V))
    for i, j in enumerate([3, 4, 5, 6, 7, 8]):
        rows[i, j] = 4.0
    masked = np.array([1, 1, 1, 1, 1, 0], np.uint8)
    prev = np.array([3, 9, -1, 6, 2, 8], np.int32)  # row 4 has a previous guess that changes
    m, tok = masked.copy(), np.full(6, -7, np.int32)
    am = prev.copy()
    _, _, st = oracle.unmask(bf_bits(rows), V, [0, 6], 1, m, tok, am)
    # rows with a previous prediction among M_t: 0,1,3,4; changed: 1 and 4
    assert st[0, 1] == 2 / 4
    assert list(am) == [3, 4, 5, 6, 7, 8]


def test_multi_request_rows_do_not_mix():
    V = 8
    rows = _logits_with_confs([0.0, 5.0, 1.0, 4.0, 2.0, 3.0], V)
    m, tok, am = state(6)
    _, com, _ = oracle.unmask(bf_bits(rows), V, [0, 3, 6], 2, m, tok, am)
    assert list(com[0]) == [1, 2]
    assert list(com[1]) == [0, 2]  # local positions of rows 3 and 5

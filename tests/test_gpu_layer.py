"""Parity of the full-layer kernels with the fp64 oracle (oracle/layer.py):
the tcgen05 GEMM and its epilogues, RMS normalization, the embedding of the
answer rows, and one whole layer.

Tolerances: each kernel computes in fp32 and rounds its output to bf16
once, so an output must lie within one bf16 rounding (2^-8 relative, two
half-ulps) of the oracle's fp64 value on the same bf16 inputs, plus the fp32
accumulation error, bounded by 1e-3 of the output's RMS; a whole layer (eight
bf16 roundings between stages) must agree to 2% relative L2."""
import numpy as np
import pytest
import torch

from helpers import bits
from oracle import layer as L

pytestmark = pytest.mark.gpu

THETA = 500000.0


def rand_bf16(shape, seed, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(shape, generator=g) * scale).to(torch.bfloat16)


def f64(t):
    return t.detach().cpu().double().numpy()


def check_close(got, ref, what=""):
    got = f64(got)
    rms = np.sqrt((ref ** 2).mean()) + 1e-30
    err = np.abs(got - ref)
    lim = np.abs(ref) * 2.0 ** -8 + 1e-3 * rms
    bad = err > lim
    assert not bad.any(), f"{what}: {int(bad.sum())} of {bad.size} outside, worst {float((err - lim).max()):.3g}"


def linear(davet, A, W, epi=0, residual=None, out_cols=None, **kw):
    M, K = A.shape
    N = W.shape[0]
    out = torch.full((M + 3, out_cols or N), float("nan"), dtype=torch.bfloat16, device="cuda")
    if residual is not None and residual is not out:
        out[:M].copy_(residual)
        residual = out
    davet.davet_linear(A, M, K, W, N, out, epi, residual, **kw)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    assert torch.isnan(out[M:].float()).all()
    return out[:M]


@pytest.mark.parametrize("M,K,N", [(1, 64, 256), (100, 256, 512), (128, 128, 256), (300, 512, 1024),
                                   (1000, 4096, 768), (257, 1024, 2560)])
def test_linear_store(davet, M, K, N):
    A = rand_bf16((M, K), M + K).cuda()
    W = rand_bf16((N, K), N + 7, K ** -0.5).cuda()
    out = linear(davet, A, W)
    check_close(out, f64(A) @ f64(W).T, f"{M}x{K}x{N}")


def test_linear_residual_in_place(davet):
    M, K, N = 333, 512, 768
    A = rand_bf16((M, K), 1).cuda()
    W = rand_bf16((N, K), 2, K ** -0.5).cuda()
    R = rand_bf16((M, N), 3).cuda()
    ref = f64(R) + f64(A) @ f64(W).T
    x = R.clone()
    davet.davet_linear(A, M, K, W, N, x, davet.EPI_RESIDUAL, x)
    torch.cuda.synchronize()
    check_close(x, ref, "residual")


def test_linear_gated_mlp(davet):
    M, K, F = 200, 256, 768
    A = rand_bf16((M, K), 4).cuda()
    Wg = rand_bf16((F, K), 5, K ** -0.5)
    Wu = rand_bf16((F, K), 6, K ** -0.5)
    # interleave in blocks of 128 rows: gate block j, then up block j
    Wgu = torch.stack([Wg.reshape(F // 128, 128, K), Wu.reshape(F // 128, 128, K)], 1).reshape(2 * F, K).cuda()
    out = linear(davet, A, Wgu, davet.EPI_SWIGLU, out_cols=F)
    a = f64(A)
    check_close(out, L.silu(a @ f64(Wg).T) * (a @ f64(Wu).T), "swiglu")


@pytest.mark.parametrize("D,H", [(128, 4), (64, 4)])
def test_linear_rotary_qkv(davet, D, H):
    HD = H * D
    K = 256
    cu = [0, 70, 71, 300, 300, 517]
    M = cu[-1]
    A = rand_bf16((M, K), 8).cuda()
    W = rand_bf16((3 * HD, K), 9, K ** -0.5).cuda()
    max_pos = 512
    tab = torch.empty((D // 2, max_pos, 2), dtype=torch.float32, device="cuda")
    davet.davet_rope_table(max_pos, D, THETA, tab)
    cu_d = torch.tensor(cu, dtype=torch.int32, device="cuda")
    out = linear(davet, A, W, davet.EPI_ROPE, cu_seqlens=cu_d, batch=len(cu) - 1, rope_cols=2 * HD, head_dim=D,
                 rope_table=tab, max_pos=max_pos)
    y = f64(A) @ f64(W).T
    pos = L.positions(cu)
    ref = np.concatenate([L.rope(y[:, :HD], pos, H, D, THETA), L.rope(y[:, HD:2 * HD], pos, H, D, THETA),
                          y[:, 2 * HD:]], axis=1)
    check_close(out, ref, "rope")
    # the table itself (frequency-major): fp32 rounding of the fp64 angles' cos and sin
    ang = L.rope_angles(np.arange(max_pos), D, THETA).T
    t = tab.cpu().double().numpy()
    assert np.abs(t[..., 0] - np.cos(ang)).max() < 1e-6 and np.abs(t[..., 1] - np.sin(ang)).max() < 1e-6


def test_rope_position_past_the_table_is_flagged(davet):
    D, H, K = 64, 4, 64
    cu = torch.tensor([0, 40], dtype=torch.int32, device="cuda")
    tab = torch.empty((D // 2, 16, 2), dtype=torch.float32, device="cuda")
    davet.davet_rope_table(16, D, THETA, tab)
    A = rand_bf16((40, K), 10).cuda()
    W = rand_bf16((3 * H * D, K), 11, K ** -0.5).cuda()
    out = torch.empty((40, 3 * H * D), dtype=torch.bfloat16, device="cuda")
    davet.davet_device_status(clear=True)
    davet.davet_linear(A, 40, K, W, 3 * H * D, out, davet.EPI_ROPE, None, cu, 1, 2 * H * D, D, tab, 16)
    torch.cuda.synchronize()
    st, flags = davet.davet_device_status(clear=True)
    assert flags & 0x4


def test_rmsnorm_rows_and_answer_rows(davet):
    C = 4096
    cu = [0, 50, 51, 200]
    resp = [7, 1, 30]
    cu_resp = np.concatenate([[0], np.cumsum(resp)]).astype(np.int32)
    x = rand_bf16((cu[-1], C), 12, 3.0).cuda()
    g = (1 + 0.1 * rand_bf16((C,), 13).float()).to(torch.bfloat16).cuda()
    out = torch.empty_like(x)
    davet.davet_rmsnorm(x, cu[-1], C, g, 1e-5, out)
    torch.cuda.synchronize()
    check_close(out, L.rmsnorm(f64(x), f64(g), 1e-5), "rmsnorm")
    R = int(cu_resp[-1])
    outa = torch.full((R + 2, C), float("nan"), dtype=torch.bfloat16, device="cuda")
    davet.davet_rmsnorm(x, R, C, g, 1e-5, outa, torch.tensor(cu, dtype=torch.int32, device="cuda"),
                        torch.from_numpy(cu_resp).cuda(), 3)
    torch.cuda.synchronize()
    rows = np.concatenate([np.arange(cu[b + 1] - resp[b], cu[b + 1]) for b in range(3)])
    check_close(outa[:R], L.rmsnorm(f64(x)[rows], f64(g), 1e-5), "rmsnorm answers")
    assert torch.isnan(outa[R:].float()).all()


def test_embed_answers_bit_exact(davet):
    V, C = 300, 256
    table = rand_bf16((V, C), 14).cuda()
    cu = torch.tensor([0, 10, 30, 31], dtype=torch.int32, device="cuda")
    resp = [4, 0, 1]
    cu_resp = torch.tensor([0, 4, 4, 5], dtype=torch.int32, device="cuda")
    tokens = torch.tensor([-1, 17, 299, -1, 5], dtype=torch.int32, device="cuda")
    x = rand_bf16((31, C), 15).cuda()
    before = bits(x).copy()
    davet.davet_embed_answers(table, V, C, tokens, 3, cu, cu_resp, 3, 5, x)
    torch.cuda.synchronize()
    got, tb = bits(x), bits(table)
    want = before.copy()
    for row, tok in zip([6, 7, 8, 9, 30], [3, 17, 299, 3, 5]):
        want[row] = tb[tok]
    assert np.array_equal(got, want)


def test_one_layer_against_the_oracle(davet):
    """A whole layer (tiny shapes: C = 256, 4 heads of 64, F = 768) on three
    packed requests, kernel by kernel as the backbone step runs it."""
    C, H, D, F = 256, 4, 64, 768
    HD = H * D
    cu = [0, 100, 101, 260]
    N = cu[-1]
    rng = np.random.default_rng(20)

    def w(shape, fan_in):
        return torch.from_numpy(rng.standard_normal(shape) / np.sqrt(fan_in)).to(torch.bfloat16)

    g1 = torch.from_numpy(1 + 0.1 * rng.standard_normal(C)).to(torch.bfloat16)
    g2 = torch.from_numpy(1 + 0.1 * rng.standard_normal(C)).to(torch.bfloat16)
    wq, wk, wv, wo = w((HD, C), C), w((HD, C), C), w((HD, C), C), w((C, HD), HD)
    wg, wu, wd = w((F, C), C), w((F, C), C), w((C, F), F)
    x0 = torch.from_numpy(rng.standard_normal((N, C))).to(torch.bfloat16)
    ref = L.layer(f64(x0), dict(g1=f64(g1), wq=f64(wq), wk=f64(wk), wv=f64(wv), wo=f64(wo), g2=f64(g2),
                                wg=f64(wg), wu=f64(wu), wd=f64(wd)), cu, H, D, THETA, 1e-5)
    dev = "cuda"
    x = x0.to(dev)
    wqkv = torch.cat([wq, wk, wv]).to(dev)
    wgu = torch.stack([wg.reshape(F // 128, 128, C), wu.reshape(F // 128, 128, C)], 1).reshape(2 * F, C).to(dev)
    cu_d = torch.tensor(cu, dtype=torch.int32, device=dev)
    tab = torch.empty((D // 2, 512, 2), dtype=torch.float32, device=dev)
    davet.davet_rope_table(512, D, THETA, tab)
    h = torch.empty((N, C), dtype=torch.bfloat16, device=dev)
    qkv = torch.empty((N, 3 * HD), dtype=torch.bfloat16, device=dev)
    att = torch.empty((N, HD), dtype=torch.bfloat16, device=dev)
    a = torch.empty((N, F), dtype=torch.bfloat16, device=dev)
    davet.davet_rmsnorm(x, N, C, g1.to(dev), 1e-5, h)
    davet.davet_linear(h, N, C, wqkv, 3 * HD, qkv, davet.EPI_ROPE, None, cu_d, 3, 2 * HD, D, tab, 512)
    davet.davet_step_attention(qkv, cu_d, 3, N, H, D, D ** -0.5, att)
    davet.davet_linear(att, N, HD, wo.to(dev), C, x, davet.EPI_RESIDUAL, x)
    davet.davet_rmsnorm(x, N, C, g2.to(dev), 1e-5, h)
    davet.davet_linear(h, N, C, wgu, 2 * F, a, davet.EPI_SWIGLU)
    davet.davet_linear(a, N, F, wd.to(dev), C, x, davet.EPI_RESIDUAL, x)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    got = f64(x)
    rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
    assert rel < 2e-2, rel


def test_large_projection_sampled_rows(davet):
    """The 8B-class QKV shape (921 rows, 4096 -> 12288) on sampled rows."""
    M, K, N = 921, 4096, 12288
    A = rand_bf16((M, K), 21).cuda()
    W = rand_bf16((N, K), 22, K ** -0.5).cuda()
    out = linear(davet, A, W)
    rows = np.random.default_rng(5).choice(M, 48, replace=False)
    rows = np.concatenate([rows, [0, 127, 128, M - 1]])
    ref = f64(A)[rows] @ f64(W).T
    check_close(out[torch.from_numpy(rows).cuda()], ref, "qkv 8B rows")


# ------------------------------------------------------------- 2-SM tiles
# Shapes with at least one wave of 256 x 256 tiles (76 CTA pairs) take the
# CTA-pair kernel; M not a multiple of 256 leaves the odd CTA of the last row
# block partly or wholly past the end.
@pytest.mark.parametrize("M,K,N", [(512, 256, 256 * 76), (600, 512, 256 * 40), (300, 128, 256 * 80)])
def test_pair_tiles_store(davet, M, K, N):
    A = rand_bf16((M, K), 60 + M).cuda()
    W = rand_bf16((N, K), 61 + K, K ** -0.5).cuda()
    out = linear(davet, A, W)
    rows = np.unique(np.concatenate([np.random.default_rng(M).choice(M, 64, replace=False), [0, 127, 128, 255, 256,
                                                                                              M - 1]]))
    check_close(out[torch.from_numpy(rows).cuda()], f64(A)[rows] @ f64(W).T, f"pair {M}x{K}x{N}")


def test_pair_tiles_residual_and_gated_mlp(davet):
    M, K = 520, 256
    N = 256 * 38
    A = rand_bf16((M, K), 70).cuda()
    W = rand_bf16((N, K), 71, K ** -0.5).cuda()
    R = rand_bf16((M, N), 72).cuda()
    x = R.clone()
    davet.davet_linear(A, M, K, W, N, x, davet.EPI_RESIDUAL, x)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    check_close(x, f64(R) + f64(A) @ f64(W).T, "pair residual")
    F = 128 * 80
    Wg = rand_bf16((F, K), 73, K ** -0.5)
    Wu = rand_bf16((F, K), 74, K ** -0.5)
    Wgu = torch.stack([Wg.reshape(F // 128, 128, K), Wu.reshape(F // 128, 128, K)], 1).reshape(2 * F, K).cuda()
    out = linear(davet, A, Wgu, davet.EPI_SWIGLU, out_cols=F)
    a = f64(A)
    check_close(out, L.silu(a @ f64(Wg).T) * (a @ f64(Wu).T), "pair swiglu")


def test_pair_tiles_rotary(davet):
    D, H, K = 128, 64, 256
    HD = H * D
    cu = [0, 300, 301, 700]
    M = cu[-1]
    A = rand_bf16((M, K), 80).cuda()
    W = rand_bf16((3 * HD, K), 81, K ** -0.5).cuda()
    tab = torch.empty((D // 2, 1024, 2), dtype=torch.float32, device="cuda")
    davet.davet_rope_table(1024, D, THETA, tab)
    out = linear(davet, A, W, davet.EPI_ROPE, cu_seqlens=torch.tensor(cu, dtype=torch.int32, device="cuda"),
                 batch=3, rope_cols=2 * HD, head_dim=D, rope_table=tab, max_pos=1024)
    y = f64(A) @ f64(W).T
    pos = L.positions(cu)
    ref = np.concatenate([L.rope(y[:, :HD], pos, H, D, THETA), L.rope(y[:, HD:2 * HD], pos, H, D, THETA),
                          y[:, 2 * HD:]], axis=1)
    check_close(out, ref, "pair rope")


# ------------------------------------------------- K split on CTA pairs
# Few rows and few column blocks (tiles on less than half of the SM pairs)
# take the split path: K slices on separate pairs, fp32 partials added in
# slice order by a second kernel that applies the epilogue.
@pytest.mark.parametrize("M,K,N,epi", [(241, 4096, 4096, 1), (200, 12288, 4096, 1), (300, 2048, 2560, 0),
                                       (241, 1024, 2048, 2)])
def test_pair_split_k(davet, M, K, N, epi):
    nbytes = davet.davet_linear_workspace_bytes(M, K, N)
    assert nbytes > 0
    ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    A = rand_bf16((M, K), 90 + M).cuda()
    W = rand_bf16((N, K), 91 + N, K ** -0.5).cuda()
    R = rand_bf16((M, N), 92).cuda() if epi == 1 else None
    outs = []
    for _ in range(2):
        out = torch.full((M + 3, N // 2 if epi == 2 else N), float("nan"), dtype=torch.bfloat16, device="cuda")
        if R is not None:
            out[:M].copy_(R)
        davet.davet_linear(A, M, K, W, N, out, epi, out if epi == 1 else None, workspace=ws)
        torch.cuda.synchronize()
        assert davet.davet_device_status() == (0, 0)
        assert torch.isnan(out[M:].float()).all()
        outs.append(out[:M].clone())
    assert torch.equal(outs[0], outs[1])
    y = f64(A) @ f64(W).T
    if epi == 0:
        ref = y
    elif epi == 1:
        ref = f64(R) + y
    else:
        F = N // 2
        blocks = y.reshape(M, F // 128, 2, 128)
        ref = (L.silu(blocks[:, :, 0]) * blocks[:, :, 1]).reshape(M, F)
    check_close(outs[0], ref, f"split {M}x{K}x{N} epi {epi}")


@pytest.mark.parametrize("D,H", [(128, 4), (64, 8)])
def test_pair_split_k_rotary(davet, D, H):
    K = 1024
    HD = H * D
    cu = [0, 37, 150, 201]
    M = cu[-1]
    A = rand_bf16((M, K), 95).cuda()
    W = rand_bf16((3 * HD, K), 96, K ** -0.5).cuda()
    tab = torch.empty((D // 2, 256, 2), dtype=torch.float32, device="cuda")
    davet.davet_rope_table(256, D, THETA, tab)
    nbytes = davet.davet_linear_workspace_bytes(M, K, 3 * HD)
    assert nbytes > 0
    ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    out = linear(davet, A, W, davet.EPI_ROPE, cu_seqlens=torch.tensor(cu, dtype=torch.int32, device="cuda"),
                 batch=3, rope_cols=2 * HD, head_dim=D, rope_table=tab, max_pos=256, workspace=ws)
    y = f64(A) @ f64(W).T
    pos = L.positions(cu)
    ref = np.concatenate([L.rope(y[:, :HD], pos, H, D, THETA), L.rope(y[:, HD:2 * HD], pos, H, D, THETA),
                          y[:, 2 * HD:]], axis=1)
    check_close(out, ref, "split rope")


def test_split_workspace_too_small_runs_one_pass(davet):
    M, K, N = 241, 4096, 4096
    A = rand_bf16((M, K), 97).cuda()
    W = rand_bf16((N, K), 98, K ** -0.5).cuda()
    out = linear(davet, A, W, workspace=torch.empty(256, dtype=torch.uint8, device="cuda"))
    check_close(out, f64(A) @ f64(W).T, "fallback")


@pytest.mark.parametrize("M,N", [(129, 256 * 76), (129, 4096), (257, 4096)])
def test_pair_tiles_single_valid_row_in_the_odd_cta(davet, M, N):
    """M = 129: the odd CTA of the pair holds one valid row (row 128); with
    N = 4096 the K split path too (its reduction sees one row of that CTA)."""
    K = 4096 if N == 4096 else 256
    A = rand_bf16((M, K), 100 + M).cuda()
    W = rand_bf16((N, K), 101, K ** -0.5).cuda()
    nbytes = davet.davet_linear_workspace_bytes(M, K, N)
    ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device="cuda")
    out = linear(davet, A, W, workspace=ws)
    rows = np.array(sorted({0, 1, 127, 128, M - 1}))
    check_close(out[torch.from_numpy(rows).cuda()], f64(A)[rows] @ f64(W).T, f"edge {M}x{K}x{N}")


# ------------------------------------------- row count read on the device
# rows_dev: the kernels are launched for a capacity of M rows and read the
# row count m from device memory when they start; rows from m on keep their
# contents, rows below m match the oracle (and, bit for bit, the launch
# without rows_dev: the tiling and the K slices are chosen for M).
@pytest.mark.parametrize("M,m,K,N,epi", [(100, 37, 256, 512, 0),      # one-CTA tiles
                                         (700, 300, 512, 1024, 1),    # CTA pairs, residual
                                         (700, 129, 512, 1024, 2),    # pairs, one valid row in the odd CTA
                                         (700, 0, 256, 512, 0),       # nothing to compute
                                         (241, 97, 4096, 4096, 1),    # pairs with the K split
                                         (241, 241, 1024, 2048, 2),   # K split, every row
                                         (500, 900, 256, 256, 0)])    # a count above M is clamped to M
def test_linear_device_row_count(davet, M, m, K, N, epi):
    A = rand_bf16((M, K), 110 + M).cuda()
    W = rand_bf16((N, K), 111 + N, K ** -0.5).cuda()
    R = rand_bf16((M, N), 112).cuda() if epi == 1 else None
    nbytes = davet.davet_linear_workspace_bytes(M, K, N)
    ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device="cuda")
    cols = N // 2 if epi == 2 else N
    outs = []
    for rows_dev in (None, torch.tensor([m], dtype=torch.int32, device="cuda")):
        out = torch.full((M, cols), -7.0, dtype=torch.bfloat16, device="cuda")
        if R is not None:
            out.copy_(R)
        davet.davet_linear(A, M, K, W, N, out, epi, out if epi == 1 else None, workspace=ws, rows_dev=rows_dev)
        torch.cuda.synchronize()
        # a count above M is clamped and flags the capacity bit
        st, flags = davet.davet_device_status(clear=True)
        assert flags == (0x2 if rows_dev is not None and m > M else 0)
        outs.append(out)
    full, dyn = outs
    n = min(m, M)
    untouched = R if epi == 1 else torch.full((M, cols), -7.0, dtype=torch.bfloat16, device="cuda")
    assert torch.equal(dyn[n:], untouched[n:])
    assert torch.equal(dyn[:n], full[:n])
    if n:
        y = f64(A[:n]) @ f64(W).T
        if epi == 0:
            ref = y
        elif epi == 1:
            ref = f64(R[:n]) + y
        else:
            blocks = y.reshape(n, N // 256, 2, 128)
            ref = (L.silu(blocks[:, :, 0]) * blocks[:, :, 1]).reshape(n, N // 2)
        check_close(dyn[:n], ref, f"rows_dev {m} of {M}")


def test_rotary_device_row_count(davet):
    """The rotary epilogue with the packed sequence shorter than the launch:
    cu_seqlens ends at the device count (as the gather leaves it)."""
    D, H, K = 128, 2, 256
    HD = H * D
    cu = [0, 150, 151, 333]
    M = 600
    A = rand_bf16((M, K), 113).cuda()
    W = rand_bf16((3 * HD, K), 114, K ** -0.5).cuda()
    tab = torch.empty((D // 2, 1024, 2), dtype=torch.float32, device="cuda")
    davet.davet_rope_table(1024, D, THETA, tab)
    cu_d = torch.tensor(cu, dtype=torch.int32, device="cuda")
    out = torch.full((M, 3 * HD), -7.0, dtype=torch.bfloat16, device="cuda")
    davet.davet_linear(A, M, K, W, 3 * HD, out, davet.EPI_ROPE, None, cu_d, 3, 2 * HD, D, tab, 1024,
                       rows_dev=cu_d[3:])
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    n = cu[-1]
    assert (out[n:].float() == -7.0).all()
    y = f64(A[:n]) @ f64(W).T
    pos = L.positions(cu)
    ref = np.concatenate([L.rope(y[:, :HD], pos, H, D, THETA), L.rope(y[:, HD:2 * HD], pos, H, D, THETA),
                          y[:, 2 * HD:]], axis=1)
    check_close(out[:n], ref, "rope rows_dev")


@pytest.mark.parametrize("m", [0, 1, 77, 200])
def test_rmsnorm_device_row_count(davet, m):
    M, C = 160, 512
    x = rand_bf16((M, C), 115).cuda()
    g = (1 + 0.1 * rand_bf16((C,), 116).float()).to(torch.bfloat16).cuda()
    out = torch.full((M, C), -7.0, dtype=torch.bfloat16, device="cuda")
    davet.davet_rmsnorm(x, M, C, g, 1e-5, out, rows_dev=torch.tensor([m], dtype=torch.int32, device="cuda"))
    torch.cuda.synchronize()
    st, flags = davet.davet_device_status(clear=True)
    assert flags == (0x2 if m > M else 0)
    n = min(m, M)
    assert (out[n:].float() == -7.0).all()
    if n:
        check_close(out[:n], L.rmsnorm(f64(x[:n]), f64(g), 1e-5), "rmsnorm rows_dev")


# ------------------------------------------- normalization folded into the product
# rmsnorm(A, g) W^T = rmsnorm(A, 1) (W diag g)^T: the call scales product row r
# by 1 / sqrt(sum of row_ss parts / K + eps); with W' = bf16(W diag g) as its
# weights the oracle is rmsnorm(A, 1) W'^T on the same bf16 operands.
@pytest.mark.parametrize("M,K,N,epi,split", [(300, 512, 768, 2, False), (100, 256, 512, 0, False),
                                             (241, 4096, 4096, 0, True), (200, 1024, 2048, 2, True)])
def test_linear_folded_rmsnorm(davet, M, K, N, epi, split):
    A = rand_bf16((M, K), 120 + M, 3.0).cuda()
    g = (1 + 0.1 * rand_bf16((K,), 121).float())
    W = rand_bf16((N, K), 122 + N, K ** -0.5)
    Wf = (W.float() * g[None, :]).to(torch.bfloat16).cuda()
    ss = torch.empty((M, 1), dtype=torch.float32, device="cuda")
    davet.davet_row_sumsq(A, M, K, ss)
    nbytes = davet.davet_linear_workspace_bytes(M, K, N)
    assert (nbytes > 0) == split
    ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device="cuda")
    out = linear(davet, A, Wf, epi, out_cols=N // 2 if epi == 2 else N, workspace=ws, row_ss=ss, row_ss_parts=1,
                 row_ss_eps=1e-5)
    y = L.rmsnorm(f64(A), np.ones(K), 1e-5) @ f64(Wf).T
    if epi == 2:
        blocks = y.reshape(M, N // 256, 2, 128)
        y = (L.silu(blocks[:, :, 0]) * blocks[:, :, 1]).reshape(M, N // 2)
    check_close(out, y, f"folded norm {M}x{K}x{N} epi {epi}")
    # the sums of squares themselves, against the fp64 sums of the bf16 rows
    assert np.allclose(ss.cpu().numpy()[:, 0], (f64(A) ** 2).sum(1), rtol=1e-5)


@pytest.mark.parametrize("M,K,N,parts_from_split", [(100, 256, 512, False), (333, 512, 768, False),
                                                    (241, 4096, 4096, True)])
def test_linear_sums_of_squares_out_feed_the_next_product(davet, M, K, N, parts_from_split):
    """A residual projection emits each row's sums of squares per 256 columns
    (ss_out); they are the sums of the stored bf16 values, and as row_ss of
    the next product they normalize its rows like rmsnorm would."""
    A = rand_bf16((M, K), 130).cuda()
    W = rand_bf16((N, K), 131, K ** -0.5).cuda()
    R = rand_bf16((M, N), 132).cuda()
    nbytes = davet.davet_linear_workspace_bytes(M, K, N)
    assert (nbytes > 0) == parts_from_split
    ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device="cuda")
    x = R.clone()
    parts = N // 256
    ss = torch.full((M, parts), float("nan"), dtype=torch.float32, device="cuda")
    davet.davet_linear(A, M, K, W, N, x, davet.EPI_RESIDUAL, x, workspace=ws, ss_out=ss)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    check_close(x, f64(R) + f64(A) @ f64(W).T, "residual with ss_out")
    xs = f64(x).reshape(M, parts, 256)
    assert np.allclose(ss.cpu().numpy(), (xs ** 2).sum(2), rtol=1e-5, atol=0)
    # the next product normalizes x's rows from those sums
    N2 = 512
    W2 = rand_bf16((N2, N), 133, N ** -0.5).cuda()
    out = linear(davet, x, W2, row_ss=ss, row_ss_parts=parts, row_ss_eps=1e-5)
    check_close(out, L.rmsnorm(f64(x), np.ones(N), 1e-5) @ f64(W2).T, "normalized by ss_out")


@pytest.mark.parametrize("M,m,K,N", [(100, 37, 256, 512), (300, 150, 512, 768), (241, 97, 4096, 4096)])
def test_norm_fold_with_device_row_count(davet, M, m, K, N):
    """Sums of squares out and the folded normalization in, with the row count
    read on the device: rows from m on keep their contents and their sums."""
    A = rand_bf16((M, K), 140 + M).cuda()
    W = rand_bf16((N, K), 141, K ** -0.5).cuda()
    R = rand_bf16((M, N), 142).cuda()
    rows_dev = torch.tensor([m], dtype=torch.int32, device="cuda")
    ws = torch.empty(max(davet.davet_linear_workspace_bytes(M, K, N), 256), dtype=torch.uint8, device="cuda")
    parts = N // 256
    x = R.clone()
    ss = torch.full((M, parts), float("nan"), dtype=torch.float32, device="cuda")
    davet.davet_linear(A, M, K, W, N, x, davet.EPI_RESIDUAL, x, workspace=ws, ss_out=ss, rows_dev=rows_dev)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    assert torch.equal(x[m:], R[m:]) and torch.isnan(ss[m:]).all()
    check_close(x[:m], f64(R[:m]) + f64(A[:m]) @ f64(W).T, "residual rows_dev")
    assert np.allclose(ss[:m].cpu().numpy(), (f64(x[:m]).reshape(m, parts, 256) ** 2).sum(2), rtol=1e-5, atol=0)
    # the next product over the same rows, normalized from those sums
    W2 = rand_bf16((512, N), 143, N ** -0.5).cuda()
    out = torch.full((M, 512), -7.0, dtype=torch.bfloat16, device="cuda")
    ws2 = torch.empty(max(davet.davet_linear_workspace_bytes(M, N, 512), 256), dtype=torch.uint8, device="cuda")
    davet.davet_linear(x, M, N, W2, 512, out, workspace=ws2, row_ss=ss, row_ss_parts=parts, row_ss_eps=1e-5,
                       rows_dev=rows_dev)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    assert (out[m:].float() == -7.0).all()
    check_close(out[:m], L.rmsnorm(f64(x[:m]), np.ones(N), 1e-5) @ f64(W2).T, "normalized rows_dev")


def test_row_sumsq_device_row_count(davet):
    M, C, m = 90, 4096, 33
    x = rand_bf16((M, C), 144, 2.0).cuda()
    ss = torch.full((M, 1), float("nan"), dtype=torch.float32, device="cuda")
    davet.davet_row_sumsq(x, M, C, ss, rows_dev=torch.tensor([m], dtype=torch.int32, device="cuda"))
    torch.cuda.synchronize()
    assert torch.isnan(ss[m:]).all()
    assert np.allclose(ss[:m, 0].cpu().numpy(), (f64(x[:m]) ** 2).sum(1), rtol=1e-5)


@pytest.mark.parametrize("m,flag", [(-3, 0x4), (250, 0x2)])
def test_device_row_count_out_of_range_is_flagged(davet, m, flag):
    """A device row count outside [0, M] is clamped (to 0 or M) and sets a bit
    of the device error word: capacity above M, argument below 0.  Covers the
    one-CTA and pair products, the RMS normalization and the sums of squares."""
    K, N = 256, 512
    rows_dev = torch.tensor([m], dtype=torch.int32, device="cuda")
    mm = min(max(m, 0), 200)
    for M in (100, 200):  # one-CTA tiles, CTA pairs
        mc = min(max(m, 0), M)
        A = rand_bf16((M, K), 150 + M).cuda()
        W = rand_bf16((N, K), 151, K ** -0.5).cuda()
        out = torch.full((M, N), -7.0, dtype=torch.bfloat16, device="cuda")
        ws = torch.empty(max(davet.davet_linear_workspace_bytes(M, K, N), 256), dtype=torch.uint8, device="cuda")
        davet.davet_device_status(clear=True)
        davet.davet_linear(A, M, K, W, N, out, workspace=ws, rows_dev=rows_dev)
        torch.cuda.synchronize()
        st, flags = davet.davet_device_status(clear=True)
        assert flags & flag, (M, m, flags)
        assert (out[mc:].float() == -7.0).all()
        if mc:
            check_close(out[:mc], f64(A[:mc]) @ f64(W[:]).T, "clamped rows_dev")
    M, C = 200, 1024
    x = rand_bf16((M, C), 152).cuda()
    g = torch.ones(C, dtype=torch.bfloat16, device="cuda")
    y = torch.full((M, C), -7.0, dtype=torch.bfloat16, device="cuda")
    davet.davet_rmsnorm(x, M, C, g, 1e-5, y, rows_dev=rows_dev)
    torch.cuda.synchronize()
    st, flags = davet.davet_device_status(clear=True)
    assert flags & flag
    assert (y[mm:].float() == -7.0).all()
    ss = torch.full((M, 1), float("nan"), dtype=torch.float32, device="cuda")
    davet.davet_row_sumsq(x, M, C, ss, rows_dev=rows_dev)
    torch.cuda.synchronize()
    st, flags = davet.davet_device_status(clear=True)
    assert flags & flag
    assert torch.isnan(ss[mm:]).all()
    if mm:
        assert np.allclose(ss[:mm, 0].cpu().numpy(), (f64(x[:mm]) ** 2).sum(1), rtol=1e-5)
    assert davet.davet_device_status() == (0, 0)

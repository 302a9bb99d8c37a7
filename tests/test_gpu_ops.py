"""Kernel-level parity on the GPU: each hot-path kernel, called through the C ABI
(include/wam_ops.h), against the oracle's arithmetic on the same bf16-representable inputs."""
import numpy as np
import pytest
import torch

from oracle import wam_oracle as O
from paper_2609_34608_gb300 import wam as W

pytestmark = pytest.mark.gpu


def _bf16(a):
    return torch.from_numpy(np.asarray(a, dtype=np.float32)).to(torch.bfloat16)


def _f64(t):
    return t.to(torch.float64).cpu().numpy()


GEMM_SHAPES = [
    (1, 128, 64), (100, 384, 128), (128, 128, 64), (129, 256, 192),
    (1296, 2304, 768),     # QKV of the 12-block d768 model, one episode
    (300, 768, 3072),      # MLP down-projection width
    (2500, 1024, 1024),
    (4914, 3456, 1152),    # QKV of the 28-block d1152 model, one episode
    (20000, 1024, 1024),   # enough tiles for the 256-wide variant
]


def _check_gemm(M, N, K, epi, run):
    """Run `run(A, Wt, bias, C, gate, rows_per_item)` on seeded bf16 operands and compare with the
    float64 product plus the epilogue's tail."""
    rng = np.random.default_rng(M * 7 + N * 3 + K + epi)
    A = _bf16(rng.standard_normal((M, K)))
    Wt = _bf16(rng.standard_normal((N, K)) * 0.05)
    bias = torch.from_numpy((rng.standard_normal(N) * 0.1).astype(np.float32))
    acc = _f64(A) @ _f64(Wt).T + bias.double().numpy()
    dev = torch.device("cuda")
    Ad, Wd, bd = A.to(dev), Wt.to(dev), bias.to(dev)
    rpi = 37
    if epi in (W.EPI_BF16, W.EPI_GELU_BF16):
        C = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device=dev)
        expect = O.gelu_tanh(acc) if epi == W.EPI_GELU_BF16 else acc
        run(Ad, Wd, bd, C, None, rpi)
        torch.cuda.synchronize()
        err = np.max(np.abs(_f64(C) - expect))
        assert err <= 8e-3 * np.max(np.abs(expect)) + 1e-3
    elif epi == W.EPI_F32:
        C = torch.full((M, N), float("nan"), dtype=torch.float32, device=dev)
        run(Ad, Wd, bd, C, None, rpi)
        torch.cuda.synchronize()
        assert np.max(np.abs(_f64(C) - acc)) <= 1e-4 * np.max(np.abs(acc))
    else:
        items = (M + rpi - 1) // rpi
        gate = torch.from_numpy(rng.standard_normal((items, N + 4)).astype(np.float32))
        h0 = torch.from_numpy(rng.standard_normal((M, N)).astype(np.float32))
        C = h0.to(dev)
        run(Ad, Wd, bd, C, gate.to(dev), rpi)
        torch.cuda.synchronize()
        g = gate.double().numpy()[np.arange(M) // rpi, :N]
        expect = h0.double().numpy() + g * acc
        assert np.max(np.abs(_f64(C) - expect)) <= 1e-4 * np.max(np.abs(expect))
    return C


@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
@pytest.mark.parametrize("epi", [W.EPI_BF16, W.EPI_GELU_BF16, W.EPI_RESID_F32, W.EPI_F32])
def test_gemm_tcgen05_matches_reference(wamlib, M, N, K, epi):
    def run(A, Wt, b, C, gate, rpi):
        W.op_gemm_bf16(A, Wt, b, C, M, N, K, epi, gate=gate, gate_stride=N + 4, rows_per_item=rpi)
    _check_gemm(M, N, K, epi, run)


# (M, N, K, tile width, K ranges): every kernel variant the planner can choose, incl. K splits.
PLAN_CASES = [
    (1392, 768, 3072, 128, 2),   # MLP down-projection widths of the 12-block d768 model (ragged M)
    (1392, 768, 768, 128, 2),    # its attention out-projection widths
    (1392, 768, 3072, 64, 1),
    (300, 768, 3072, 64, 4),
    (129, 256, 192, 128, 3),     # K = 192: one-atom stages, three ranges, ragged M
    (1392, 3072, 768, 256, 1),
    (200, 512, 768, 128, 3),     # three ranges: the partials fill the stage buffers exactly
    (1, 128, 256, 128, 2),       # a single row, two ranges of one stage each
]


@pytest.mark.parametrize("M,N,K,tile_n,k_splits", PLAN_CASES)
@pytest.mark.parametrize("epi", [W.EPI_BF16, W.EPI_GELU_BF16, W.EPI_RESID_F32, W.EPI_F32])
def test_gemm_plans_match_reference(wamlib, M, N, K, tile_n, k_splits, epi):
    ws = torch.zeros(W.gemm_workspace_bytes(), dtype=torch.uint8, device="cuda")

    def run(A, Wt, b, C, gate, rpi):
        W.op_gemm_bf16_plan(A, Wt, b, C, M, N, K, epi, tile_n, k_splits, workspace=ws, gate=gate,
                            gate_stride=N + 4, rows_per_item=rpi)
    _check_gemm(M, N, K, epi, run)
    # the ticket counters are back at zero for the next call
    n_sms = torch.cuda.get_device_properties(0).multi_processor_count
    assert int(ws[ws.numel() - 4 * n_sms:].count_nonzero()) == 0


# (M, N, K, tile width): shapes where the two-CTA clusters apply (even column-tile count)
CLUSTER_CASES = [(1296, 768, 768, 64), (1296, 3072, 768, 128), (1296, 768, 3072, 64), (1296, 2304, 768, 128),
                 (129, 256, 256, 128), (1, 256, 128, 64), (2600, 1024, 1024, 64)]


@pytest.mark.parametrize("M,N,K,tile_n", CLUSTER_CASES)
@pytest.mark.parametrize("epi", [W.EPI_GELU_BF16, W.EPI_RESID_F32])
def test_gemm_clusters_match_reference_and_single_ctas(wamlib, M, N, K, tile_n, epi):
    """Clusters of two CTAs sharing the A tile by multicast: the reference within tolerance, and the
    single-CTA kernel bit for bit (same accumulation order)."""
    outs = []
    for cluster in (2, 1):
        def run(A, Wt, b, C, gate, rpi):
            W.op_gemm_bf16_plan(A, Wt, b, C, M, N, K, epi, tile_n, 1, gate=gate, gate_stride=N + 4,
                                rows_per_item=rpi, cluster=cluster)
        outs.append(_check_gemm(M, N, K, epi, run).cpu())
    assert torch.equal(outs[0], outs[1])


# (M, N, K, tile width) for CTA pairs on one 256-row MMA: the projections of one episode of the
# 12-block d768 model (the second CTA of the last pair holds only rows past M), a single row, a
# ragged M with 128-wide pair tiles, and enough units that each pair runs several tiles (both
# TMEM accumulators in turn, the second CTA releasing them to the first).
PAIR_CASES = [(1296, 3072, 768, 256), (1296, 2304, 768, 256), (1296, 768, 768, 128), (1, 256, 128, 256),
              (129, 512, 256, 128), (20000, 1024, 1024, 256)]


@pytest.mark.parametrize("M,N,K,tile_n", PAIR_CASES)
@pytest.mark.parametrize("epi", [W.EPI_BF16, W.EPI_GELU_BF16, W.EPI_RESID_F32, W.EPI_F32])
def test_gemm_cta_pairs_match_reference_and_single_ctas(wamlib, M, N, K, tile_n, epi):
    """Two-SM MMA pairs (tcgen05 cta_group::2): the reference within tolerance, and the single-CTA
    kernel of the same tile width bit for bit (the same K order into the fp32 accumulator)."""
    outs = []
    for cluster in (3, 1):
        def run(A, Wt, b, C, gate, rpi):
            W.op_gemm_bf16_plan(A, Wt, b, C, M, N, K, epi, tile_n, 1, gate=gate, gate_stride=N + 4,
                                rows_per_item=rpi, cluster=cluster)
        outs.append(_check_gemm(M, N, K, epi, run).cpu())
    assert torch.equal(outs[0], outs[1])


def test_gemm_split_is_deterministic(wamlib):
    """A K-split result does not depend on which unit finished last: repeated runs agree bit for bit."""
    M, N, K = 1392, 768, 3072
    rng = np.random.default_rng(5)
    dev = torch.device("cuda")
    A = _bf16(rng.standard_normal((M, K))).to(dev)
    Wt = _bf16(rng.standard_normal((N, K)) * 0.05).to(dev)
    ws = torch.zeros(W.gemm_workspace_bytes(), dtype=torch.uint8, device=dev)
    outs = []
    for _ in range(3):
        C = torch.empty((M, N), dtype=torch.float32, device=dev)
        W.op_gemm_bf16_plan(A, Wt, None, C, M, N, K, W.EPI_F32, 128, 2, workspace=ws)
        outs.append(C.cpu())
    assert all(torch.equal(outs[0], o) for o in outs[1:])


def test_gemm_plan_rejections(wamlib):
    dev = torch.device("cuda")
    A = torch.zeros((1392, 768), dtype=torch.bfloat16, device=dev)
    Wt = torch.zeros((768, 768), dtype=torch.bfloat16, device=dev)
    C = torch.zeros((1392, 768), dtype=torch.float32, device=dev)
    ws = torch.zeros(W.gemm_workspace_bytes(), dtype=torch.uint8, device=dev)
    with pytest.raises(W.WamError):   # a split without a workspace
        W.op_gemm_bf16_plan(A, Wt, None, C, 1392, 768, 768, W.EPI_F32, 128, 2)
    with pytest.raises(W.WamError):   # 6 K stages do not split in 4
        W.op_gemm_bf16_plan(A, Wt, None, C, 1392, 768, 768, W.EPI_F32, 128, 4, workspace=ws)
    with pytest.raises(W.WamError):   # 11 x 12 x 2 units exceed one wave
        W.op_gemm_bf16_plan(A, Wt, None, C, 1392, 768, 768, W.EPI_F32, 64, 2, workspace=ws)
    with pytest.raises(W.WamError):   # no such tile width
        W.op_gemm_bf16_plan(A, Wt, None, C, 1392, 768, 768, W.EPI_F32, 96, 1, workspace=ws)
    with pytest.raises(W.WamError):   # 256-wide partials of two ranges exceed the stage buffers
        W.op_gemm_bf16_plan(A[:200], Wt, None, C[:200], 200, 768, 768, W.EPI_F32, 256, 2, workspace=ws)
    with pytest.raises(W.WamError):   # CTA pairs never split K
        W.op_gemm_bf16_plan(A, Wt, None, C, 1392, 768, 768, W.EPI_F32, 128, 2, workspace=ws, cluster=3)
    with pytest.raises(W.WamError):   # CTA pairs take 128- or 256-wide tiles
        W.op_gemm_bf16_plan(A, Wt, None, C, 1392, 768, 768, W.EPI_F32, 64, 1, cluster=3)
    with pytest.raises(W.WamError):   # no such cluster mode
        W.op_gemm_bf16_plan(A, Wt, None, C, 1392, 768, 768, W.EPI_F32, 128, 1, cluster=4)


def test_gemm_rejects_unsupported_shapes(wamlib):
    dev = torch.device("cuda")
    A = torch.zeros((4, 96), dtype=torch.bfloat16, device=dev)
    Wt = torch.zeros((128, 96), dtype=torch.bfloat16, device=dev)
    C = torch.zeros((4, 128), dtype=torch.bfloat16, device=dev)
    with pytest.raises(W.WamError):
        W.op_gemm_bf16(A, Wt, None, C, 4, 128, 96, W.EPI_BF16)


@pytest.mark.parametrize("M,N,K", [(1, 64, 16), (77, 130, 45), (300, 512, 128)])
def test_gemm_f32_matches_reference(wamlib, M, N, K):
    rng = np.random.default_rng(M + N + K)
    A = rng.standard_normal((M, K)).astype(np.float32)
    Wt = rng.standard_normal((N, K)).astype(np.float32)
    b = rng.standard_normal(N).astype(np.float32)
    dev = torch.device("cuda")
    C = torch.empty((M, N), dtype=torch.float32, device=dev)
    W.op_gemm_f32(torch.from_numpy(A).to(dev), torch.from_numpy(Wt).to(dev), torch.from_numpy(b).to(dev), C,
                  M, N, K, W.EPI_F32)
    torch.cuda.synchronize()
    ref = A.astype(np.float64) @ Wt.astype(np.float64).T + b
    assert np.max(np.abs(C.cpu().numpy() - ref)) <= 1e-5 * np.max(np.abs(ref)) * np.sqrt(K)


ATTN_CASES = [
    (1, 1, 2, 64), (1, 56, 2, 64), (2, 64, 2, 64), (1, 100, 3, 64), (2, 1296, 2, 64),
    (1, 65, 2, 72), (1, 257, 2, 72), (1, 4914, 1, 72),
]


@pytest.mark.parametrize("B,N,H,dh", ATTN_CASES)
def test_attention_bf16_matches_oracle(wamlib, B, N, H, dh):
    rng = np.random.default_rng(B * 1000 + N + H + dh)
    d = H * dh
    qkv = _bf16(rng.standard_normal((B * N, 3 * d)))
    dev = torch.device("cuda")
    out = torch.full((B * N, d), float("nan"), dtype=torch.bfloat16, device=dev)
    W.op_attention(qkv.to(dev), out, B, N, d, H, "bf16")
    torch.cuda.synchronize()
    q64 = _f64(qkv)
    got = _f64(out)
    for b in range(B):
        blk = q64[b * N:(b + 1) * N]
        ref = O.attention(blk[:, :d], blk[:, d:2 * d], blk[:, 2 * d:], H)
        assert np.max(np.abs(got[b * N:(b + 1) * N] - ref)) <= 2e-2


def test_attention_f32_matches_oracle(wamlib):
    rng = np.random.default_rng(9)
    B, N, H, dh = 2, 56, 4, 32
    d = H * dh
    qkv = rng.standard_normal((B * N, 3 * d)).astype(np.float32)
    dev = torch.device("cuda")
    out = torch.empty((B * N, d), dtype=torch.float32, device=dev)
    W.op_attention(torch.from_numpy(qkv).to(dev), out, B, N, d, H, "fp32")
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    for b in range(B):
        blk = qkv[b * N:(b + 1) * N].astype(np.float64)
        ref = O.attention(blk[:, :d], blk[:, d:2 * d], blk[:, 2 * d:], H)
        assert np.max(np.abs(got[b * N:(b + 1) * N] - ref)) <= 2e-5


@pytest.mark.parametrize("prec,d", [("bf16", 768), ("fp32", 128), ("bf16", 1152)])
def test_ln_modulate_matches_oracle(wamlib, prec, d):
    rng = np.random.default_rng(d)
    M, rpi = 300, 100
    h = (rng.standard_normal((M, d)) * 3 + 0.5).astype(np.float32)
    mods = (rng.standard_normal((M // rpi, 2 * d)) * 0.3).astype(np.float32)
    dev = torch.device("cuda")
    md = torch.from_numpy(mods).to(dev)
    out = torch.empty((M, d), dtype=torch.bfloat16 if prec == "bf16" else torch.float32, device=dev)
    W.op_ln_modulate(torch.from_numpy(h).to(dev), md.data_ptr(), md.data_ptr() + 4 * d, 2 * d, out, M, d, rpi, prec)
    torch.cuda.synchronize()
    item = np.arange(M) // rpi
    ref = O.layer_norm(h.astype(np.float64)) * (1 + mods[item, d:]) + mods[item, :d]
    tol = 1e-2 if prec == "bf16" else 2e-5
    assert np.max(np.abs(_f64(out) - ref)) <= tol * np.max(np.abs(ref))


TC_ATTN_CASES = [(1, 1, 2, 64), (1, 56, 2, 64), (2, 128, 2, 64), (1, 129, 4, 64), (1, 1296, 12, 64),
                 (2, 300, 2, 64), (1, 2464, 4, 64), (2, 2464, 16, 64), (8, 600, 8, 64), (20, 130, 8, 64),
                 # head dim 72 (the bimanual model: 16 heads, d 1152), ragged and multi-item
                 (1, 1, 16, 72), (1, 200, 16, 72), (2, 130, 16, 72), (1, 4914, 16, 72), (3, 600, 16, 72)]


@pytest.mark.parametrize("B,N,H,dh", TC_ATTN_CASES)
def test_attention_tcgen05_matches_oracle(wamlib, B, N, H, dh):
    """QKV projection writing V^T, then the tcgen05 attention, against the oracle's attention of
    the same bf16 q, k, v."""
    rng = np.random.default_rng(B * 100 + N + H + dh)
    d = dh * H
    dev = torch.device("cuda")
    x = _bf16(rng.standard_normal((B * N, d)))
    Wt = _bf16(rng.standard_normal((3 * d, d)) / np.sqrt(d))
    bias = torch.from_numpy((rng.standard_normal(3 * d) * 0.1).astype(np.float32))
    vt_ld = (N + 7) // 8 * 8
    qkv = torch.full((B * N, 3 * d), float("nan"), dtype=torch.bfloat16, device=dev)
    vt = torch.zeros((B * d, vt_ld), dtype=torch.bfloat16, device=dev)
    out = torch.full((B * N, d), float("nan"), dtype=torch.bfloat16, device=dev)
    W.op_gemm_qkv_vt(x.to(dev), Wt.to(dev), bias.to(dev), qkv, vt, B * N, d, N, vt_ld)
    W.op_attention_tc(qkv, vt, out, B, N, d, H)
    torch.cuda.synchronize()
    proj = torch.from_numpy(_f64(x) @ _f64(Wt).T + bias.double().numpy())
    qk = _f64(qkv)[:, :2 * d]
    assert np.max(np.abs(qk - proj.numpy()[:, :2 * d])) <= 2e-2 * np.max(np.abs(proj.numpy()))
    v_from_vt = _f64(vt).reshape(B, H, dh, vt_ld)[..., :N].transpose(0, 3, 1, 2).reshape(B * N, d)
    assert np.max(np.abs(v_from_vt - proj.numpy()[:, 2 * d:])) <= 2e-2 * np.max(np.abs(proj.numpy()))
    got = _f64(out)
    for b in range(B):
        blk = slice(b * N, (b + 1) * N)
        ref = O.attention(qk[blk, :d], qk[blk, d:], v_from_vt[blk], H)
        assert np.max(np.abs(got[blk] - ref)) <= 2e-2

"""Each hot-path kernel through the C ABI (featfix_ops.h) against the oracle
or the plain definition, on seeded inputs spanning several tiles and a
ragged tail."""

import numpy as np
import pytest
import torch

import oracle
from paper_2607_27842_gb300 import featfix as ff

from .gpu_helpers import rel_l2

pytestmark = pytest.mark.gpu

TD = {"f32": torch.float32, "bf16": torch.bfloat16}


def randn(shape, dtype, seed, scale=1.0, dev="cuda"):
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    return (torch.randn(shape, generator=g) * scale).to(TD[dtype]).to(dev)


def f64(t):
    return t.detach().to("cpu", torch.float64).numpy()


# ----------------------------------------------------------------------------
# draft (Eq. 2)
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("K", [0, 1, 2, 3])
def test_draft_exact_on_polynomial_increments(cuda, K):
    """Order-K draft reproduces degree-K increment trajectories (fp32 mode)."""
    n = 3 * 4096 + 7                         # several CTAs of vectors + a scalar tail
    s = [40, 33, 25, 12][:K + 1]
    g = torch.Generator().manual_seed(K)
    coef = torch.randn((K + 1, n), generator=g, dtype=torch.float64) * 0.1
    traj = lambda t: sum(coef[d] * (float(t) / 40.0) ** d for d in range(K + 1))
    hist = [traj(si).to(torch.float32).to(cuda) for si in s]
    t = 47
    _, _, w = ff.featfix_plan_build(t + 1, 1, sorted(set(s) | {0}), K, ())
    x = randn(n, "f32", 9)
    u = f64(x)
    ff.featfix_op_draft("f32", x, hist, w[t, :K + 1])
    torch.cuda.synchronize()
    want = u + traj(t).numpy()
    assert rel_l2(f64(x) - u, want - u) < 1e-5


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("n", [5 * 8192 + 24, 29831168 + 24])   # small; HunyuanVideo's E (tensors > L2) + tail
def test_draft_matches_oracle(cuda, dtype, n):
    s = [18, 12, 6]
    hist = [randn(n, dtype, 10 + j, 0.05) for j in range(3)]
    x = randn(n, dtype, 3)
    u = f64(x)
    _, _, w = ff.featfix_plan_build(20, 1, [0, 6, 12, 18], 2, ())
    ff.featfix_op_draft(dtype, x, hist, w[20 - 1, :3])
    torch.cuda.synchronize()
    ref = oracle.draft.draft(u, [(s[j], f64(hist[j])) for j in range(3)], 19, 2)
    tol = 1e-6 if dtype == "f32" else 4e-3
    assert rel_l2(f64(x), ref) < tol


# ----------------------------------------------------------------------------
# paid check + forward (Eqs. 3-5)
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("n", [1000, 4718592 + 8, 29831168 + 8])   # tiny, DiT-XL/2's E, HunyuanVideo's E
def test_verify_sums_and_forwarding(cuda, dtype, n):
    hist = [randn(n, dtype, 20 + j, 0.05) for j in range(2)]
    w = [1.4, -0.4]
    u = randn(n, dtype, 30)
    hf = (u.float() + randn(n, "f32", 31, 0.05)).to(TD[dtype])
    ws = torch.empty(ff.featfix_op_verify_workspace(n), dtype=torch.uint8, device=cuda)
    sums = torch.zeros(4, dtype=torch.float64, device=cuda)
    u_keep = u.clone()
    ff.featfix_op_verify(dtype, u, hist, w, hf, sums, ws, write_draft=False)
    torch.cuda.synchronize()
    assert torch.equal(u, u_keep)
    # h_d as the draft kernel stores it
    hd = u_keep.clone()
    ff.featfix_op_draft(dtype, hd, hist, w)
    torch.cuda.synchronize()
    d = f64(hd) - f64(hf)
    f = f64(hf)
    want = [np.abs(d).sum(), np.abs(f).sum(), (d * d).sum(), (f * f).sum()]
    np.testing.assert_allclose(sums.cpu().numpy(), want, rtol=2e-5)
    # Verify arm: u is overwritten by exactly the drafted tensor
    sums2 = torch.zeros(4, dtype=torch.float64, device=cuda)
    ff.featfix_op_verify(dtype, u, hist, w, hf, sums2, ws, write_draft=True)
    torch.cuda.synchronize()
    assert torch.equal(u, hd)
    assert torch.equal(sums, sums2)          # deterministic reduction order


def test_verify_rejects_small_workspace(cuda):
    n = 1 << 20
    x = torch.zeros(n, device=cuda)
    ws = torch.empty(8, dtype=torch.uint8, device=cuda)
    sums = torch.zeros(4, dtype=torch.float64, device=cuda)
    with pytest.raises(ff.FeatFixError) as e:
        ff.featfix_op_verify("f32", x, [x], [1.0], x, sums, ws)
    assert e.value.status == ff.ERR_INVALID_ARG


# ----------------------------------------------------------------------------
# LayerNorm + modulation
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("dtype,C,rows,rpb", [("f32", 128, 300, 100), ("bf16", 1152, 300, 100),
                                              ("bf16", 3072, 300, 100),
                                              ("bf16", 2048, 14310, 14310)])   # HunyuanVideo image stream
def test_ln_modulate(cuda, dtype, C, rows, rpb):
    x = randn((rows, C), dtype, 1, 2.0)
    mod = randn(((rows + rpb - 1) // rpb, 2 * C), "f32", 2, 0.1)
    out = torch.empty_like(x)
    ff.featfix_op_ln_modulate(dtype, x, out, rows, C, mod[:, :C], mod[:, C:], 2 * C, rpb)
    torch.cuda.synchronize()
    xm = f64(x)
    m = f64(mod)
    b = np.arange(rows) // rpb
    ref = oracle.model.layer_norm(xm) * (1 + m[b, C:]) + m[b, :C]
    assert rel_l2(f64(out), ref) < (1e-6 if dtype == "f32" else 4e-3)


# ----------------------------------------------------------------------------
# dense layers with the fused epilogue
# ----------------------------------------------------------------------------

GEMM_SHAPES = [
    (256, 256, 128),      # one tile of each width
    (300, 200, 1152),     # ragged M and N
    (130, 32, 64),        # final projection width
    (512, 3456, 1152),    # DiT-XL/2 qkv width, several N tiles
    (4096, 1152, 4608),   # DiT-XL/2 fc2, full size
    (4096, 4608, 1152),   # DiT-XL/2 fc1, full size
    (14310, 6144, 2048),  # HunyuanVideo image-stream qkv, full size
    (14310, 2048, 8192),  # HunyuanVideo image-stream fc2 (K = 8192: CTA-pair tiles), full size
]


@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_gemm_plain_and_bias(cuda, dtype, M, N, K):
    if dtype == "f32" and M * N * K > 1e9:
        pytest.skip("CUDA-core path is checked on small shapes")
    a = randn((M, K), dtype, 1)
    w = randn((N, K), dtype, 2, 0.05)
    bias = randn(N, dtype, 3)
    out = torch.empty((M, N), dtype=TD[dtype], device=cuda)
    ff.featfix_op_gemm(dtype, a, w, out, bias=bias)
    torch.cuda.synchronize()
    if M * N * K > 1e11:     # large shapes: a sample of rows against the plain definition
        r = np.unique(np.linspace(0, M - 1, 700).astype(int))
        ref = f64(a)[r] @ f64(w).T + f64(bias)
        assert rel_l2(f64(out)[r], ref) < 5e-3
        return
    ref = f64(a) @ f64(w).T + f64(bias)
    tol = 1e-5 if dtype == "f32" else 5e-3
    assert rel_l2(f64(out), ref) < tol


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("M,N,K,rpb", [(384, 256, 192, 128),      # row-wise epilogue
                                       (1100, 520, 192, 500),     # ragged: a swapped tile of 8 columns
                                       (4096, 1152, 1152, 256),   # DiT-XL/2 out-projection: 4 x 32 + 16 swapped tiles
                                       (512, 2048, 8192, 256)])   # K = 8192: CTA-pair tiles, staged epilogue
def test_gemm_fused_epilogues(cuda, dtype, M, N, K, rpb):
    a = randn((M, K), dtype, 4)
    w = randn((N, K), dtype, 5, 0.08)
    bias = randn(N, dtype, 6, 0.3)
    gate = randn(((M + rpb - 1) // rpb, 2 * N), "f32", 7)
    resid = randn((M, N), dtype, 8)
    out = torch.empty((M, N), dtype=TD[dtype], device=cuda)
    hout = torch.empty_like(out)
    ff.featfix_op_gemm(dtype, a, w, out, bias=bias, act=1, gate=gate[:, N:], gate_stride=2 * N, rows_per_batch=rpb,
                       resid=resid, hist_base=resid, hist_out=hout)
    torch.cuda.synchronize()
    y = oracle.model.gelu_tanh(f64(a) @ f64(w).T + f64(bias))
    b = np.arange(M) // rpb
    ref = f64(resid) + f64(gate)[b, N:] * y
    tol = 1e-5 if dtype == "f32" else 5e-3
    assert rel_l2(f64(out), ref) < tol
    # history increment = stored output - base, computed from the stored value
    inc = f64(out) - f64(resid)
    assert rel_l2(f64(hout), inc) < (1e-6 if dtype == "f32" else 4e-3)


def test_gemm_is_deterministic(cuda):
    a = randn((1024, 1152), "bf16", 11)
    w = randn((3456, 1152), "bf16", 12, 0.05)
    o1 = torch.empty((1024, 3456), dtype=torch.bfloat16, device=cuda)
    o2 = torch.empty_like(o1)
    ff.featfix_op_gemm("bf16", a, w, o1)
    ff.featfix_op_gemm("bf16", a, w, o2)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2)


# ----------------------------------------------------------------------------
# attention over the joint [text ; image] sequence
# ----------------------------------------------------------------------------

ATTN_CASES = [
    # dtype, B, n_txt, n_img, heads, d
    ("bf16", 2, 0, 256, 3, 72),
    # at most two key tiles, head width <= 80: K / V resident, one N = 256 S
    ("bf16", 4, 0, 100, 3, 72),        # one key tile (N = 128 S), ragged
    ("bf16", 2, 40, 60, 2, 72),        # text tile + image tile, both ragged
    ("bf16", 2, 5, 100, 2, 64),        # head width 64 (no tail box)
    ("bf16", 3, 0, 256, 5, 64),
    ("bf16", 1, 5, 70, 2, 128),
    ("bf16", 2, 3, 130, 2, 64),
    ("bf16", 1, 0, 200, 4, 32),
    ("f32", 1, 0, 64, 4, 32),
    ("f32", 2, 7, 40, 2, 72),
    # longer sequences: ragged text / image tails, several query and key
    # tiles (an odd number of query tiles), the tensor-core head widths
    ("bf16", 2, 77, 1000, 2, 128),
    ("bf16", 1, 0, 1100, 3, 72),
    ("bf16", 2, 130, 1030, 2, 64),
    # full-size attention of two workloads: DiT-XL/2 (256 image tokens, 16
    # heads x 72, model batch 16) and FLUX (512 text + 4096 image tokens,
    # 24 heads x 128)
    ("bf16", 16, 0, 256, 16, 72),
    ("bf16", 1, 512, 4096, 24, 128),
    # HunyuanVideo: 256 text + 14310 video tokens, 16 heads x 128
    ("bf16", 1, 256, 14310, 16, 128),
]


def short_items_per_cta(nt, ni, B, H):
    """Query tiles one CTA takes in turn on short sequences (at most four
    key tiles): as few as keep all CTAs within one wave of two per SM."""
    nq = (nt + 127) // 128 + (ni + 127) // 128
    if nq > 4:
        return 0
    slots = 2 * torch.cuda.get_device_properties(0).multi_processor_count
    ipc = 1
    while ipc < nq and -(-nq // ipc) * B * H > slots:
        ipc += 1
    return ipc


# short sequences whose CTAs walk several query tiles: (B, n_txt, n_img, heads,
# d, items per CTA on a 152-SM GPU, what the case exercises)
MULTI_ITEM_CASES = [
    (8, 0, 300, 16, 72, 2, "3 query tiles in CTAs of 2: the last CTA's second item is dead"),
    (16, 0, 300, 16, 72, 3, "3 items per CTA"),
    (16, 5, 300, 16, 72, 4, "4 items per CTA, the first a 5-token text tile"),
    (8, 9, 300, 12, 64, 2, "text + ragged image tiles, 2 items per CTA, both CTAs whole"),
]


@pytest.mark.parametrize("B,nt,ni,H,d,want,what", MULTI_ITEM_CASES, ids=[c[-1][:24] for c in MULTI_ITEM_CASES])
def test_attention_multi_item_ctas(cuda, B, nt, ni, H, d, want, what):
    ipc = short_items_per_cta(nt, ni, B, H)
    if ipc != want:
        pytest.skip("this GPU's SM count gives %d items per CTA, the case is built for %d" % (ipc, want))
    test_attention_matches_oracle(cuda, "bf16", B, nt, ni, H, d)


@pytest.mark.parametrize("dtype,B,nt,ni,H,d", ATTN_CASES)
def test_attention_matches_oracle(cuda, dtype, B, nt, ni, H, d):
    C = H * d
    T = B * (nt + ni)
    ld = 3 * C + 16                            # row stride wider than q|k|v
    qkv = randn((T, ld), dtype, 13)
    out = torch.zeros((T, C + 8), dtype=TD[dtype], device=cuda)
    ff.featfix_op_attention(dtype, qkv, out, B, nt, ni, H, d)
    torch.cuda.synchronize()
    rows = np.array([[b * nt + n if n < nt else B * nt + b * ni + (n - nt) for n in range(nt + ni)]
                     for b in range(B)])
    Q = f64(qkv)[rows]
    q = Q[..., :C].reshape(B, nt + ni, H, d).transpose(0, 2, 1, 3)
    k = Q[..., C:2 * C].reshape(B, nt + ni, H, d).transpose(0, 2, 1, 3)
    v = Q[..., 2 * C:3 * C].reshape(B, nt + ni, H, d).transpose(0, 2, 1, 3)
    got = f64(out)[rows][..., :C].reshape(B, nt + ni, H, d)
    # long sequences: the float64 score matrix of every head would not fit,
    # so the first, a middle and the last head are checked
    heads = range(H) if B * H * (nt + ni) ** 2 <= 5e7 else sorted({0, H // 2, H - 1})
    for h in heads:
        ref = oracle.model.attention(q[:, h:h + 1], k[:, h:h + 1], v[:, h:h + 1])[:, 0]
        assert rel_l2(got[:, :, h], ref) < (1e-5 if dtype == "f32" else 1e-2), h
    assert np.all(f64(out)[:, C:] == 0)        # nothing written past C

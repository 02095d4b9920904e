"""Pins of the CPU oracle against what the paper and mathematics fix.

Each test checks oracle code against something other than itself: a library
routine, brute force, a closed form, a published test vector, or one of the
invariants the paper states for FeatFix (Eq. 5 "by construction", the
Exact-only audit, the Verify control, accounting).  A plausible slip in the
oracle (dropped term, wrong sign, swapped index or operand) fails one of them.
"""

import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import draft, featfix, flops, model, noise, sampler, schedule
from paper_2607_27842_gb300 import synthetic

from .conftest import golden_lines

RNG = np.random.default_rng(1234)


def rnd(*shape, scale=1.0):
    return RNG.standard_normal(shape) * scale


def t64(a):
    return torch.from_numpy(np.ascontiguousarray(a))


# ----------------------------------------------------------------------------
# primitives vs library routines and brute force
# ----------------------------------------------------------------------------

def test_layer_norm_matches_torch():
    x = rnd(3, 5, 48, scale=3.0) + 1.5
    ref = F.layer_norm(t64(x), (48,), eps=1e-6).numpy()
    np.testing.assert_allclose(model.layer_norm(x), ref, rtol=1e-12, atol=1e-12)


def test_gelu_and_silu_match_torch():
    x = rnd(1000, scale=4.0)
    np.testing.assert_allclose(model.gelu_tanh(x), F.gelu(t64(x), approximate="tanh").numpy(), rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(model.silu(x), F.silu(t64(x)).numpy(), rtol=1e-12, atol=1e-14)


def test_linear_is_nn_linear():
    x, w, b = rnd(4, 7), rnd(5, 7), rnd(5)
    np.testing.assert_allclose(model.linear(x, w, b), F.linear(t64(x), t64(w), t64(b)).numpy(), rtol=1e-12)


def test_attention_matches_sdpa_and_brute_force():
    q, k, v = rnd(2, 3, 9, 8), rnd(2, 3, 9, 8), rnd(2, 3, 9, 8)
    out = model.attention(q, k, v)
    ref = F.scaled_dot_product_attention(t64(q), t64(k), t64(v)).numpy()
    np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-12)
    # brute force, one query at a time, softmax written out
    b, h, i = 1, 2, 4
    scores = [sum(q[b, h, i, e] * k[b, h, j, e] for e in range(8)) / math.sqrt(8) for j in range(9)]
    ex = [math.exp(s) for s in scores]
    z = sum(ex)
    o = [sum(ex[j] / z * v[b, h, j, e] for j in range(9)) for e in range(8)]
    np.testing.assert_allclose(out[b, h, i], o, rtol=1e-10)


def test_heads_split_is_contiguous_per_head():
    x = np.arange(2 * 3 * 12, dtype=np.float64).reshape(2, 3, 12)
    s = model.split_heads(x, 4)
    assert s.shape == (2, 4, 3, 3)
    np.testing.assert_array_equal(s[1, 2, 0], x[1, 0, 6:9])
    np.testing.assert_array_equal(model.merge_heads(s), x)


# ----------------------------------------------------------------------------
# rotary embedding
# ----------------------------------------------------------------------------

def test_rope_is_complex_rotation():
    x = rnd(1, 2, 5, 16)
    ang = rnd(5, 8)
    out = model.apply_rope(x, ang)
    z = (x[..., 0::2] + 1j * x[..., 1::2]) * np.exp(1j * ang)
    np.testing.assert_allclose(out[..., 0::2], z.real, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(out[..., 1::2], z.imag, rtol=1e-12, atol=1e-12)


def test_rope_scores_depend_on_relative_position_only():
    d = 16
    axes = (8, 8)
    q, k = rnd(d), rnd(d)
    def score(pq, pk):
        aq = model.rope_angles(np.array([pq]), axes)
        ak = model.rope_angles(np.array([pk]), axes)
        rq = model.apply_rope(q[None, None, None], aq)[0, 0, 0]
        rk = model.apply_rope(k[None, None, None], ak)[0, 0, 0]
        return rq @ rk
    assert abs(score((3, 5), (1, 2)) - score((7, 9), (5, 6))) < 1e-10
    assert abs(score((0, 0), (0, 0)) - q @ k) < 1e-12


def test_rope_axes_and_frequencies():
    assert model.rope_axes(128, 2) == (64, 64)
    assert model.rope_axes(128, 3) == (16, 56, 56)
    ang = model.rope_angles(np.array([[2, 5]]), (4, 4))
    np.testing.assert_allclose(ang[0], [2.0, 2.0 * 10000 ** -0.5, 5.0, 5.0 * 10000 ** -0.5])


def test_patch_grid_and_image_positions_row_major():
    """The image tokens' grid positions: last axis fastest (2-D: row, column;
    3-D: frame, row, column), written out by hand for small grids, and the
    grids of the video and image workloads."""
    np.testing.assert_array_equal(model.image_positions((2, 3)),
                                  [[0, 0], [0, 1], [0, 2], [1, 0], [1, 1], [1, 2]])
    np.testing.assert_array_equal(model.image_positions((2, 1, 2)),
                                  [[0, 0, 0], [0, 0, 1], [1, 0, 0], [1, 0, 1]])
    assert model.patch_grid(synthetic.SHAPES["hunyuan"]) == ((9, 30, 53), 4)
    assert model.patch_grid(synthetic.SHAPES["flux"]) == ((64, 64), 4)
    assert model.patch_grid(synthetic.SHAPES["dit_xl2"]) == ((16, 16), 4)


def test_rope_table_of_a_video_token():
    """3-D rotary angles of one image token (frame 2, row 1, column 4 of a
    3 x 2 x 5 grid, token 2*10 + 1*5 + 4 = 29): the 16 / 56 / 56 axis split of
    a 128-wide head, pair j of an axis of width w turning by
    position * 10000^(-2j / w)."""
    sh = synthetic.reduced(synthetic.SHAPES["hunyuan"], lat_f=3, lat_h=4, lat_w=10)
    ang = model.rope_table(sh)
    assert ang.shape == (30, 64)
    a = ang[29]
    for off, width, pos in ((0, 16, 2.0), (8, 56, 1.0), (36, 56, 4.0)):
        for j in range(width // 2):
            assert a[off + j] == pytest.approx(pos * 10000.0 ** (-2.0 * j / width), rel=1e-12)
    assert model.rope_table(synthetic.SHAPES["dit_xl2"]) is None


# ----------------------------------------------------------------------------
# embeddings and layout
# ----------------------------------------------------------------------------

def test_timestep_sinusoid_closed_form():
    s0 = model.timestep_sinusoid(0.0)
    np.testing.assert_array_equal(s0[:128], 1.0)
    np.testing.assert_array_equal(s0[128:], 0.0)
    s = model.timestep_sinusoid(3.0)
    assert s[0] == pytest.approx(math.cos(3.0)) and s[128] == pytest.approx(math.sin(3.0))
    assert s[64] == pytest.approx(math.cos(3.0 * 10000 ** -0.5))


def test_sincos_position_closed_form():
    C, gh, gw = 16, 3, 4
    pe = model.sincos_pos_2d(C, gh, gw)
    np.testing.assert_allclose(pe[0], [0, 0, 0, 0, 1, 1, 1, 1] * 2)
    tok = 1 * gw + 2  # row 1, column 2
    np.testing.assert_allclose(pe[tok, 0], math.sin(1.0))
    np.testing.assert_allclose(pe[tok, 1], math.sin(10000 ** -0.25))
    np.testing.assert_allclose(pe[tok, 8], math.sin(2.0))
    np.testing.assert_allclose(pe[tok, 12], math.cos(2.0))


def test_patchify_layout_and_inverse():
    sh = synthetic.reduced(synthetic.SHAPES["dit_xl2"], lat_h=4, lat_w=6, batch=2, in_ch=3, out_ch=3)
    x = rnd(2, 3, 4, 6)
    p = model.patchify(x, sh)
    assert p.shape == (2, 6, 12)
    # token (1, 2) of sample 1, feature (channel 2, row offset 1, col offset 0)
    assert p[1, 1 * 3 + 2, 2 * 4 + 1 * 2 + 0] == x[1, 2, 1 * 2 + 1, 2 * 2 + 0]
    np.testing.assert_array_equal(model.unpatchify(p, sh, 3), x)
    shv = synthetic.reduced(synthetic.SHAPES["hunyuan"], lat_f=2, lat_h=4, lat_w=4, in_ch=2, out_ch=2, patch_t=1)
    xv = rnd(1, 2, 2, 4, 4)
    pv = model.patchify(xv, shv)
    assert pv.shape == (1, 8, 8)
    assert pv[0, 1 * 4 + 1 * 2 + 1, 1 * 4 + 0 * 2 + 1] == xv[0, 1, 1, 2, 3]
    np.testing.assert_array_equal(model.unpatchify(pv, shv, 2), xv)


# ----------------------------------------------------------------------------
# blocks (Eq. 1) vs torch.nn.functional compositions and structural cases
# ----------------------------------------------------------------------------

def small_dit(**kw):
    base = dict(n_dual=2, hidden=32, heads=4, head_dim=8, mlp=64, in_ch=4, out_ch=8, patch=2, lat_h=8, lat_w=8,
                n_classes=5, batch=2, cfg=True, dtype="f32", sampler="ddim")
    base.update(kw)
    return synthetic.reduced(synthetic.SHAPES["dit_xl2"], **base)


def small_mmdit(**kw):
    base = dict(n_dual=2, n_single=2, hidden=32, heads=2, head_dim=16, mlp=64, in_ch=4, out_ch=4, patch=2, lat_h=8,
                lat_w=8, txt_tokens=5, batch=1, cfg=False, dtype="f32", rope_dims=2)
    base.update(kw)
    return synthetic.reduced(synthetic.SHAPES["flux"], **base)


def weights64(shape, seed=0, scale=1.0):
    w = synthetic.oracle_weights(synthetic.make_weights(shape, seed=seed))
    return {k: v * scale for k, v in w.items()}


def torch_dit_block(W, pre, u, c, heads):
    u, c = t64(u), t64(c)
    T = {k: t64(v) for k, v in W.items() if k.startswith(pre)}
    m = F.linear(F.silu(c), T[pre + "mod.w"], T[pre + "mod.b"]).chunk(6, dim=-1)
    B, N, C = u.shape
    a = F.layer_norm(u, (C,), eps=1e-6) * (1 + m[1][:, None]) + m[0][:, None]
    qkv = F.linear(a, T[pre + "qkv.w"], T[pre + "qkv.b"]).reshape(B, N, 3, heads, C // heads).permute(2, 0, 3, 1, 4)
    o = F.scaled_dot_product_attention(qkv[0], qkv[1], qkv[2]).transpose(1, 2).reshape(B, N, C)
    u1 = u + m[2][:, None] * F.linear(o, T[pre + "proj.w"], T[pre + "proj.b"])
    a2 = F.layer_norm(u1, (C,), eps=1e-6) * (1 + m[4][:, None]) + m[3][:, None]
    y = F.linear(F.gelu(F.linear(a2, T[pre + "fc1.w"], T[pre + "fc1.b"]), approximate="tanh"), T[pre + "fc2.w"],
                 T[pre + "fc2.b"])
    return (u1 + m[5][:, None] * y).numpy()


def test_dit_block_matches_torch_composition():
    sh = small_dit()
    W = weights64(sh, scale=10.0)  # larger weights: every term matters
    u = rnd(4, 16, 32)
    c = rnd(4, 32)
    out = model.exact_block(W, sh, 1, u, c)
    np.testing.assert_allclose(out, torch_dit_block(W, "blk1.", u, c, 4), rtol=1e-10, atol=1e-10)


def test_zero_gates_make_every_block_the_identity():
    sh = small_mmdit()
    W = weights64(sh, scale=10.0)
    C = sh.hidden
    for name in list(W):
        if name.endswith("mod.w") or name.endswith("mod.b"):
            if name.startswith("single"):
                W[name][2 * C:3 * C] = 0.0
            elif name.startswith("dual"):
                W[name][2 * C:3 * C] = 0.0
                W[name][5 * C:6 * C] = 0.0
    u = rnd(1, sh.tokens, C)
    c = rnd(1, C)
    for l in range(sh.n_layers):
        np.testing.assert_array_equal(model.exact_block(W, sh, l, u, c), u)
    shd = small_dit()
    Wd = weights64(shd)
    for l in range(shd.n_dual):
        Wd["blk%d.mod.w" % l][2 * 32:3 * 32] = 0.0
        Wd["blk%d.mod.b" % l][2 * 32:3 * 32] = 0.0
        Wd["blk%d.mod.w" % l][5 * 32:6 * 32] = 0.0
        Wd["blk%d.mod.b" % l][5 * 32:6 * 32] = 0.0
    ud = rnd(4, 16, 32)
    np.testing.assert_array_equal(model.exact_block(Wd, shd, 0, ud, rnd(4, 32)), ud)


def test_dual_block_without_text_is_the_dit_block():
    sh = small_mmdit(txt_tokens=0, rope_dims=0)
    W = weights64(sh, scale=5.0)
    u, c = rnd(1, sh.img_tokens, 32), rnd(1, 32)
    Wd = {"b." + k.split("img_")[1]: v for k, v in W.items() if k.startswith("dual0.img_")}
    ref = model.dit_block(Wd, "b.", u, c, sh.heads)
    np.testing.assert_allclose(model.exact_block(W, sh, 0, u, c), ref, rtol=1e-12, atol=1e-12)


def test_dual_block_streams_use_their_own_weights():
    """Perturbing a text-stream weight moves image tokens only through attention."""
    sh = small_mmdit(rope_dims=0)
    W = weights64(sh, scale=5.0)
    u, c = rnd(1, sh.tokens, 32), rnd(1, 32)
    base = model.exact_block(W, sh, 0, u, c)
    W2 = dict(W)
    W2["dual0.txt_fc2.b"] = W["dual0.txt_fc2.b"] + 1.0
    out = model.exact_block(W2, sh, 0, u, c)
    np.testing.assert_array_equal(out[:, 5:], base[:, 5:])
    assert np.abs(out[:, :5] - base[:, :5]).max() > 1e-3


def torch_rope(z, ang, n_txt):
    """Rotary embedding on tokens >= n_txt as complex multiplication."""
    rot = torch.polar(torch.ones_like(t64(ang)), t64(ang))
    zi = z[:, :, n_txt:]
    zc = torch.view_as_complex(zi.reshape(*zi.shape[:-1], zi.shape[-1] // 2, 2).contiguous()) * rot
    return torch.cat([z[:, :, :n_txt], torch.view_as_real(zc).reshape(zi.shape)], dim=2)


def test_dual_block_matches_torch_composition():
    sh = small_mmdit(batch=2)
    W = weights64(sh, scale=5.0)
    u, c = rnd(2, sh.tokens, 32), rnd(2, 32)
    ang = model.rope_table(sh)
    out = model.exact_block(W, sh, 1, u, c, ang)
    T = {k: t64(v) for k, v in W.items() if k.startswith("dual1.")}
    tu, tc = t64(u), t64(c)
    nt = sh.txt_tokens

    def ln_mod(x, sh_, sc_):
        return F.layer_norm(x, (32,), eps=1e-6) * (1 + sc_[:, None]) + sh_[:, None]

    mods = {s: F.linear(F.silu(tc), T["dual1.%s_mod.w" % s], T["dual1.%s_mod.b" % s]).chunk(6, -1)
            for s in ("img", "txt")}
    parts = {"txt": tu[:, :nt], "img": tu[:, nt:]}
    qkv = torch.cat([F.linear(ln_mod(parts[s], mods[s][0], mods[s][1]), T["dual1.%s_qkv.w" % s],
                              T["dual1.%s_qkv.b" % s]) for s in ("txt", "img")], dim=1)
    q, k, v = (z.reshape(2, sh.tokens, 2, 16).transpose(1, 2) for z in qkv.chunk(3, dim=-1))
    o = F.scaled_dot_product_attention(torch_rope(q, ang, nt), torch_rope(k, ang, nt), v)
    o = o.transpose(1, 2).reshape(2, sh.tokens, 32)
    outs = []
    for s, osl in (("txt", o[:, :nt]), ("img", o[:, nt:])):
        m = mods[s]
        x = parts[s] + m[2][:, None] * F.linear(osl, T["dual1.%s_proj.w" % s], T["dual1.%s_proj.b" % s])
        y = F.linear(F.gelu(F.linear(ln_mod(x, m[3], m[4]), T["dual1.%s_fc1.w" % s], T["dual1.%s_fc1.b" % s]),
                            approximate="tanh"), T["dual1.%s_fc2.w" % s], T["dual1.%s_fc2.b" % s])
        outs.append(x + m[5][:, None] * y)
    np.testing.assert_allclose(out, torch.cat(outs, dim=1).numpy(), rtol=1e-10, atol=1e-10)


def test_single_block_matches_torch_composition():
    sh = small_mmdit()
    W = weights64(sh, scale=5.0)
    u, c = rnd(1, sh.tokens, 32), rnd(1, 32)
    ang = model.rope_table(sh)
    out = model.exact_block(W, sh, 2, u, c, ang)
    T = {k: t64(v) for k, v in W.items() if k.startswith("single0.")}
    tu, tc = t64(u), t64(c)
    sh_, sc_, g_ = F.linear(F.silu(tc), T["single0.mod.w"], T["single0.mod.b"]).chunk(3, dim=-1)
    a = F.layer_norm(tu, (32,), eps=1e-6) * (1 + sc_[:, None]) + sh_[:, None]
    y = F.linear(a, T["single0.lin1.w"], T["single0.lin1.b"])
    qkv, mlp = y[..., :96], y[..., 96:]
    q, k, v = (z.reshape(1, sh.tokens, 2, 16).transpose(1, 2) for z in qkv.chunk(3, dim=-1))
    # rotary on image tokens via complex multiplication
    rot = torch.polar(torch.ones_like(t64(ang)), t64(ang))
    def rope(z):
        zi = z[:, :, 5:]
        zc = torch.view_as_complex(zi.reshape(*zi.shape[:-1], 8, 2).contiguous()) * rot
        return torch.cat([z[:, :, :5], torch.view_as_real(zc).reshape(zi.shape)], dim=2)
    o = F.scaled_dot_product_attention(rope(q), rope(k), v).transpose(1, 2).reshape(1, sh.tokens, 32)
    ref = tu + g_[:, None] * F.linear(torch.cat([o, F.gelu(mlp, approximate="tanh")], -1), T["single0.lin2.w"],
                                      T["single0.lin2.b"])
    np.testing.assert_allclose(out, ref.numpy(), rtol=1e-10, atol=1e-10)


# ----------------------------------------------------------------------------
# draft (Eq. 2)
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("K", [0, 1, 2, 3])
def test_order_k_draft_is_exact_on_degree_k_trajectories(K):
    s = [23, 17, 12, 4][:K + 1]          # uneven refresh spacing, newest first
    coef = rnd(K + 1, 6)
    def traj(t):
        return sum(coef[d] * float(t) ** d for d in range(K + 1))
    hist = [(si, traj(si)) for si in s]
    for t in (24, 26, 30):
        u = rnd(6)
        out = draft.draft(u, hist, t, K)
        np.testing.assert_allclose(out, u + traj(t), rtol=1e-9, atol=1e-9)


def test_order_zero_is_reuse():
    hist = [(8, rnd(5)), (4, rnd(5))]
    u = rnd(5)
    np.testing.assert_array_equal(draft.draft(u, hist, 11, 0), u + hist[0][1])


def test_first_order_weights_closed_form_and_partition_of_unity():
    s0, s1, t = 12, 6, 15
    e0, e1 = np.array([1.0, 0.0]), np.array([0.0, 1.0])
    w0 = draft.taylor_forecast(t, [s0, s1], [e0, e0 * 0])[0]
    w1 = draft.taylor_forecast(t, [s0, s1], [e1 * 0, e1])[1]
    dlt = (t - s0) / (s0 - s1)
    assert w0 == pytest.approx(1 + dlt) and w1 == pytest.approx(-dlt)
    for K in (1, 2, 3):
        s = [20, 15, 9, 2][:K + 1]
        ones = [np.ones(1) for _ in s]
        assert draft.taylor_forecast(27, s, ones)[0] == pytest.approx(1.0)


def test_second_order_taylor_equals_lagrange_basis():
    s, t = [10, 5, 0], 13
    for j in range(3):
        R = [np.array([1.0 if m == j else 0.0]) for m in range(3)]
        lag = np.prod([(t - s[m]) / (s[j] - s[m]) for m in range(3) if m != j])
        assert draft.taylor_forecast(t, s, R)[0] == pytest.approx(lag)


def test_recursive_variant_error_on_quadratics():
    """Uniform spacing d, R(t) = c t^2: the recursive estimator's forecast
    misses by -c d (t - s0) (backward differences estimate the derivative at
    s0 - d/2); it equals the interpolant for K = 1."""
    c, d = 0.7, 5
    s = [20, 15, 10]
    hist = [(si, np.array([c * si * si])) for si in s]
    for t in (22, 24):
        rec = draft.draft(np.zeros(1), hist, t, 2, variant="recursive")[0]
        assert rec == pytest.approx(c * t * t - c * d * (t - s[0]))
        lin_r = draft.draft(np.zeros(1), hist[:2], t, 1, variant="recursive")[0]
        lin_i = draft.draft(np.zeros(1), hist[:2], t, 1)[0]
        assert lin_r == pytest.approx(lin_i)


# ----------------------------------------------------------------------------
# schedule (Section 3.3)
# ----------------------------------------------------------------------------

def test_tiny_plan_matches_hand_derivation():
    wl = synthetic.workload("tiny")
    kind, keff = schedule.build_plan(wl.steps, 4, wl.refresh, wl.K, wl.sites, "featfix")
    letters = {schedule.EXACT: "E", schedule.DRAFT: "D", schedule.SITE: "S"}
    for line in golden_lines("plan_tiny.txt"):
        i, ks, ke = line.split()[:3]
        i = int(i)
        assert "".join(letters[k] for k in kind[i]) == ks
        if int(ke) >= 0:
            assert keff[i] == int(ke)


@pytest.mark.parametrize("bad", [
    dict(refresh=(1, 3)),                       # step 0 not a refresh
    dict(sites=((3, 0),)),                      # site on a refresh step
    dict(sites=((4, 9),)),                      # layer out of range
    dict(sites=((4, 1), (4, 1))),               # duplicate site
    dict(K=4),                                  # order out of range
    dict(refresh=(0, 0, 3)),                    # duplicate refresh
    dict(refresh=(0, 10)),                      # refresh out of range
])
def test_schedule_rules(bad):
    args = dict(steps=10, L=4, refresh=(0, 3, 6, 9), K=1, sites=((4, 2),))
    args.update(bad)
    with pytest.raises(schedule.ScheduleError):
        schedule.build_plan(args["steps"], args["L"], args["refresh"], args["K"], args["sites"], "featfix")


def test_history_entries_by_hand():
    """The refresh steps a draft reads (newest first, at most K + 1 = 2) on
    the tiny schedule (refreshes 0, 3, 6, 9; sites (4, 2), (7, 1)), written
    out from Section 3.3's rules: refreshes push every block; a site pushes
    its own block only with the site-history reading (reading 5)."""
    steps, L, ref, K, sites = 10, 4, (0, 3, 6, 9), 1, ((4, 2), (7, 1))
    h = schedule.block_history_steps(steps, L, ref, K, sites, "featfix")
    assert h[0] == [None] * 4 and h[3] == [None] * 4
    assert h[1] == [[0]] * 4 and h[2] == [[0]] * 4
    assert h[4] == [[3, 0]] * 4                  # the site (4, 2) drafts from the same entries
    assert h[5][2] == [3, 0] and h[8] == [[6, 3]] * 4
    hs = schedule.block_history_steps(steps, L, ref, K, sites, "featfix", site_updates_history=True)
    assert hs[4][2] == [3, 0] and hs[5][2] == [4, 3] and hs[5][1] == [3, 0]
    assert hs[7][1] == [6, 3] and hs[8][1] == [7, 6]
    assert hs[7][2] == [6, 4] and hs[8][2] == [6, 4]  # the site's entry 4 outlives refresh 3
    assert schedule.block_history_steps(steps, L, ref, K, sites, "vanilla")[5] == [None] * 4


def test_vanilla_plan_is_all_exact():
    kind, _ = schedule.build_plan(6, 3, (0, 3), 1, ((1, 1),), "vanilla")
    assert all(k == schedule.EXACT for row in kind for k in row)


def test_diagonal_sites_avoid_refresh_steps():
    for name in ("dit_xl2", "flux", "qwen", "hunyuan"):
        wl = synthetic.workload(name)
        schedule.validate(wl.steps, wl.shape.n_layers, wl.refresh, wl.K, wl.sites)
    assert synthetic.workload("dit_xl2").sites[:3] == ((3, 1), (9, 5), (16, 8))


# ----------------------------------------------------------------------------
# samplers
# ----------------------------------------------------------------------------

def test_euler_is_exact_on_straight_paths():
    x0, noise_ = rnd(3, 4), rnd(3, 4)
    x = noise_.copy()
    N = 10
    for i in range(N):
        x = sampler.euler_update(x, noise_ - x0, N, i)
    np.testing.assert_allclose(x, x0, rtol=1e-12, atol=1e-12)


def test_ddim_recovers_data_from_true_noise():
    ab = sampler.ddim_alpha_bar()
    assert ab[0] == pytest.approx(1 - 1e-4)
    N = 50
    ts = sampler.ddim_timesteps(N)
    assert ts[0] == 980 and ts[-1] == 0
    x0, eps = rnd(2, 5), rnd(2, 5)
    x = np.sqrt(ab[ts[0]]) * x0 + np.sqrt(1 - ab[ts[0]]) * eps
    for i in range(N):
        x = sampler.ddim_update(x, eps, N, i)
    np.testing.assert_allclose(x, x0, rtol=1e-9, atol=1e-9)


def test_model_time_fed_to_the_embedding():
    """Euler: t_i = 1000 sigma_i with sigma_i = 1 - i / N (1000 at the first
    step, 1000 / N at the last); DDIM: the visited timestep 1000 - 20 (i + 1)
    at N = 50.  Straight-path exactness and DDIM recovery hold for any time
    map, so the map itself is pinned here."""
    assert sampler.model_time("euler", 50, 0) == 1000.0
    assert sampler.model_time("euler", 50, 49) == pytest.approx(20.0)
    assert sampler.model_time("euler", 10, 5) == pytest.approx(500.0)
    for i in (0, 7, 49):
        assert sampler.model_time("ddim", 50, i) == 1000 - 20 * (i + 1)
    sig = sampler.euler_sigmas(4)
    np.testing.assert_allclose(sig, [1.0, 0.75, 0.5, 0.25, 0.0])


def test_guidance_limits():
    out = rnd(4, 3)
    np.testing.assert_allclose(sampler.guide(out, 2, True, 1.0), out[:2])
    np.testing.assert_allclose(sampler.guide(out, 2, True, 0.0), out[2:])


# ----------------------------------------------------------------------------
# seeded latent
# ----------------------------------------------------------------------------

def test_splitmix64_published_sequence():
    want = [int(v) for v in golden_lines("splitmix64_seed1234567.txt")]
    assert [int(v) for v in noise.splitmix64_words(1234567, 5)] == want


def test_box_muller_moments():
    z = noise.normals(7, 400001).astype(np.float64)
    assert abs(z.mean()) < 0.01 and abs(z.std() - 1) < 0.01
    assert abs(((z ** 3).mean())) < 0.02 and abs((z ** 4).mean() - 3) < 0.05


# ----------------------------------------------------------------------------
# the sampling loop: FeatFix invariants stated in the paper
# ----------------------------------------------------------------------------

def tiny_setup():
    wl = synthetic.workload("tiny")
    sh = wl.shape
    W = synthetic.oracle_weights(synthetic.make_weights(sh, seed=0))
    cond = synthetic.oracle_cond(sh, synthetic.make_cond(sh, seed=2))
    xT = noise.initial_latent(1, sh)
    return wl, sh, W, cond, xT


def test_all_refresh_schedule_is_vanilla_bitwise():
    wl, sh, W, cond, xT = tiny_setup()
    a, _, ca = featfix.run(W, sh, cond, xT, wl.steps, list(range(wl.steps)), wl.K, (), "featfix")
    b, _, cb = featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, wl.K, wl.sites, "vanilla")
    np.testing.assert_array_equal(a, b)
    assert ca["refresh_steps"] == cb["refresh_steps"] == wl.steps


def test_identity_blocks_make_every_arm_vanilla_bitwise():
    """With every block the identity (both gates zero), the residual
    increments a refresh stores are exactly zero, so every draft is exactly
    its incoming state and every arm reproduces vanilla sampling bit for bit;
    forecasting the block outputs themselves instead of their increments
    (reading 1) would not."""
    wl, sh, W, cond, xT = tiny_setup()
    C = sh.hidden
    W = dict(W)
    for name in list(W):
        if name.startswith("blk") and (name.endswith("mod.w") or name.endswith("mod.b")):
            W[name] = W[name].copy()
            W[name][2 * C:3 * C] = 0.0
            W[name][5 * C:6 * C] = 0.0
    ref, _, _ = featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, wl.K, wl.sites, "vanilla")
    for mode in ("featfix", "verify"):
        x, logs, _ = featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, wl.K, wl.sites, mode)
        np.testing.assert_array_equal(x, ref)
        assert all(g["rel_l1"] == 0.0 and g["rel_l2"] == 0.0 for g in logs)


def test_featfix_site_forwards_the_exact_output():
    wl, sh, W, cond, xT = tiny_setup()
    seen = []
    def hook(i, l, kind, u, h, extra):
        if kind == schedule.SITE:
            hf = featfix.block_at(W, sh, l, i, wl.steps, u, cond)
            np.testing.assert_array_equal(h, hf)
            assert featfix.rel_l1(h, hf) == 0.0
            seen.append((i, l))
    featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, wl.K, wl.sites, "featfix", hook=hook)
    assert seen == sorted(wl.sites)


def test_exact_only_equals_featfix_bitwise():
    wl, sh, W, cond, xT = tiny_setup()
    a, la, ca = featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, wl.K, wl.sites, "featfix")
    b, lb, cb = featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, wl.K, wl.sites, "exact_only")
    np.testing.assert_array_equal(a, b)
    assert len(la) == 2 and lb == []
    assert ca == cb == {"refresh_steps": 4, "paid_checks": 2, "forwarded": 2}


def test_verify_forwards_the_draft_and_matches_no_sites():
    wl, sh, W, cond, xT = tiny_setup()
    v, lv, cv = featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, wl.K, wl.sites, "verify")
    n, _, _ = featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, wl.K, (), "featfix")
    np.testing.assert_array_equal(v, n)
    assert cv == {"refresh_steps": 4, "paid_checks": 2, "forwarded": 0}
    assert [(e["step"], e["layer"]) for e in lv] == [(4, 2), (7, 1)]
    assert all(e["rel_l1"] > 0 and e["rel_l2"] > 0 for e in lv)


def test_featfix_and_verify_agree_until_the_first_site_then_differ():
    wl, sh, W, cond, xT = tiny_setup()
    trace = {}
    def rec(tag):
        def hook(i, l, kind, u, h, extra):
            trace.setdefault(tag, []).append((i, l, h.copy()))
        return hook
    a, la, _ = featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, wl.K, wl.sites, "featfix", hook=rec("f"))
    b, lb, _ = featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, wl.K, wl.sites, "verify", hook=rec("v"))
    for (i, l, hf), (_, _, hv) in zip(trace["f"], trace["v"]):
        if (i, l) == (4, 2):
            break
        np.testing.assert_array_equal(hf, hv)
    # the first paid check sees the same state in both arms: same logged value
    assert la[0]["rel_l1"] == lb[0]["rel_l1"]
    assert np.abs(a - b).max() > 0


def test_site_history_push_reading():
    """SITE_UPDATES_HISTORY reading: with reuse (K = 0) a block's next draft
    after its site adds exactly the site's exact increment h_f - u; by
    default it adds the last refresh increment.  A site's own draft and
    logged discrepancy do not depend on the reading."""
    wl, sh, W, cond, xT = tiny_setup()
    (i0, l0) = sorted(wl.sites)[0]
    nxt = i0 + 1
    assert nxt not in wl.refresh
    for push in (False, True):
        inc = {}
        def hook(i, l, kind, u, h, extra):
            if l == l0 and kind != schedule.DRAFT or (l == l0 and i == nxt):
                inc[(i, kind)] = ((extra["h_f"] if extra else h) - u, h - u)
        _, logs, _ = featfix.run(W, sh, cond, xT, wl.steps, wl.refresh, 0, wl.sites, "verify", hook=hook,
                                 site_updates_history=push)
        draft_inc = inc[(nxt, schedule.DRAFT)][1]
        site_exact = inc[(i0, schedule.SITE)][0]
        last_ref = max(r for r in wl.refresh if r < i0)
        refresh_inc = inc[(last_ref, schedule.EXACT)][0]
        # (h - u recovers the added increment up to the rounding of u + R)
        want = site_exact if push else refresh_inc
        np.testing.assert_allclose(draft_inc, want, rtol=0, atol=1e-15)
        assert np.abs(site_exact - refresh_inc).max() > 0
        if not push:
            base = logs
    assert logs[0]["rel_l1"] == base[0]["rel_l1"]


def test_partial_forwarding_arms_reduce_to_the_whole_block_arms():
    """Token / channel partial forwarding: all selected = FeatFix, none
    selected = the draft (Verify's forward), and a mixed mask forwards h_f
    exactly on the selected tokens / channels of each site."""
    wl, sh, W, cond, xT = tiny_setup()
    args = (W, sh, cond, xT, wl.steps, wl.refresh, wl.K, wl.sites)
    ff_x, _, _ = featfix.run(*args, "featfix")
    vf_x, _, _ = featfix.run(*args, "verify")
    n_tok, C = sh.tokens, sh.hidden
    for axis, n in (("tokens", n_tok), ("channels", C)):
        a, _, _ = featfix.run(*args, "featfix", forward_mask=(axis, np.ones(n)))
        np.testing.assert_array_equal(a, ff_x)
        b, _, _ = featfix.run(*args, "featfix", forward_mask=(axis, np.zeros(n)))
        np.testing.assert_array_equal(b, vf_x)
        m = (np.arange(n) % 3) == 0
        seen = []
        def hook(i, l, kind, u, h, extra):
            if kind == schedule.SITE:
                sel = m[None, :, None] if axis == "tokens" else m[None, None, :]
                sel = np.broadcast_to(sel, h.shape)
                np.testing.assert_array_equal(h[sel], extra["h_f"][sel])
                np.testing.assert_array_equal(h[~sel], extra["h_d"][~sel])
                seen.append((i, l))
        c, _, _ = featfix.run(*args, "featfix", hook=hook, forward_mask=(axis, m))
        assert seen == sorted(wl.sites)
        assert np.abs(c - ff_x).max() > 0 and np.abs(c - vf_x).max() > 0


def test_discrepancy_definitions():
    hf = np.array([1.0, -2.0, 3.0])
    hd = np.array([1.5, -2.0, 2.0])
    assert featfix.rel_l1(hd, hf) == pytest.approx(1.5 / 6.0)
    assert featfix.rel_l2(hd, hf) == pytest.approx(math.sqrt(1.25) / math.sqrt(14.0))


def test_flop_counter_matches_table_1():
    """Table 1: FLUX Vanilla, 50 steps, 3734.6 TFLOPs -> 74.69 T per step; the
    19 dual + 38 single block stack at 4096 + 512 tokens gives 74.36 T (blocks
    only, within 0.5%)."""
    per_step = flops.step_flops(synthetic.SHAPES["flux"])
    assert per_step / 1e12 == pytest.approx(74.36, abs=0.01)
    assert abs(per_step / 1e12 / (3734.6 / 50) - 1) < 0.005


# ----------------------------------------------------------------------------
# conditioning, token embedding, output head and the sampler's use of the
# head (Eq. 1's conditioning c, Section 3.1's samplers)
# ----------------------------------------------------------------------------

def torch_cond(W, t, labels, batch):
    """c = Linear(SiLU(Linear(sinusoid(t)))) + label row, written with
    torch.nn.functional and torch's own sinusoid."""
    half = 128
    freqs = torch.exp(-math.log(10000.0) * torch.arange(half, dtype=torch.float64) / half)
    s = torch.cat([torch.cos(t * freqs), torch.sin(t * freqs)])
    T = {k: t64(v) for k, v in W.items()}
    e = F.linear(F.silu(F.linear(s, T["t_fc1.w"], T["t_fc1.b"])), T["t_fc2.w"], T["t_fc2.b"])
    c = e[None].expand(batch, -1)
    if labels is not None:
        c = c + F.embedding(torch.as_tensor(labels), T["y_emb"])
    return c.numpy()


def test_cond_vector_matches_torch_composition():
    sh = small_dit()
    W = weights64(sh, seed=3, scale=20.0)       # large enough that SiLU is far from linear
    labels = np.array([1, 4, 5, 5])              # the guidance half uses the null class 5
    np.testing.assert_allclose(model.cond_vector(W, 437.0, labels=labels, batch=4),
                               torch_cond(W, 437.0, labels, 4), rtol=1e-12, atol=1e-12)
    Wm = weights64(small_mmdit(), seed=3, scale=20.0)
    np.testing.assert_allclose(model.cond_vector(Wm, 12.5, batch=2), torch_cond(Wm, 12.5, None, 2),
                               rtol=1e-12, atol=1e-12)


def test_cond_vector_label_and_time_parts_separate():
    """A zero label table leaves the time MLP alone, identical for every
    sample; a zero time MLP output leaves exactly the label rows (so the
    labels are added after the MLP, never fed through it)."""
    sh = small_dit()
    W = weights64(sh, seed=5, scale=10.0)
    labels = np.array([0, 3, 5, 2])
    Wy0 = dict(W, y_emb=np.zeros_like(W["y_emb"]))
    c = model.cond_vector(Wy0, 250.0, labels=labels, batch=4)
    h = model.silu(model.timestep_sinusoid(250.0) @ W["t_fc1.w"].T + W["t_fc1.b"])
    np.testing.assert_allclose(c, np.tile(h @ W["t_fc2.w"].T + W["t_fc2.b"], (4, 1)), rtol=1e-12, atol=1e-13)
    Wt0 = dict(W, **{"t_fc2.w": np.zeros_like(W["t_fc2.w"]), "t_fc2.b": np.zeros_like(W["t_fc2.b"])})
    np.testing.assert_array_equal(model.cond_vector(Wt0, 250.0, labels=labels, batch=4), W["y_emb"][labels])


def test_embed_tokens_dit_unit_impulse():
    """One latent element set to 1: only its patch token moves, by the
    column of the patch-embedding weight its (channel, row, column) offset
    selects; every token carries bias + its 2-D sin-cos position."""
    sh = small_dit(lat_h=8, lat_w=6)
    W = weights64(sh, seed=7)
    x = np.zeros((4, sh.in_ch, 8, 6))
    x[1, 2, 5, 3] = 1.0
    tok = model.embed_tokens(W, sh, x)
    gw = 6 // 2
    n_hot = (5 // 2) * gw + 3 // 2
    f_hot = 2 * 4 + (5 % 2) * 2 + (3 % 2)
    base = W["x_emb.b"][None, None] + model.sincos_pos_2d(sh.hidden, 4, gw)[None]
    want = np.broadcast_to(base, tok.shape).copy()
    want[1, n_hot] += W["x_emb.w"][:, f_hot]
    np.testing.assert_allclose(tok, want, rtol=1e-13, atol=1e-13)


def test_embed_tokens_mmdit_text_first_no_position():
    """MMDiT: the text tokens come first, unchanged; the image tokens are
    the patch embedding alone (positions enter through the rotary
    embedding inside the blocks, not here)."""
    sh = small_mmdit(lat_f=2, lat_h=4, lat_w=6, patch_t=1, rope_dims=3, head_dim=16)
    W = weights64(sh, seed=9)
    x = np.zeros((1, sh.in_ch, 2, 4, 6))
    x[0, 3, 1, 2, 5] = 1.0
    txt = rnd(1, sh.txt_tokens, sh.hidden)
    tok = model.embed_tokens(W, sh, x, txt=txt)
    assert tok.shape == (1, sh.txt_tokens + 2 * 2 * 3, sh.hidden)
    np.testing.assert_array_equal(tok[:, :sh.txt_tokens], txt)
    img = tok[:, sh.txt_tokens:]
    n_hot = 1 * (2 * 3) + (2 // 2) * 3 + 5 // 2
    f_hot = 3 * 4 + (2 % 2) * 2 + (5 % 2)
    want = np.broadcast_to(W["img_in.b"], img.shape).copy()
    want[0, n_hot] += W["img_in.w"][:, f_hot]
    np.testing.assert_allclose(img, want, rtol=1e-13, atol=1e-13)


def torch_final(W, sh, tok, c):
    T = {k: t64(v) for k, v in W.items()}
    img = t64(tok)[:, sh.txt_tokens:] if sh.arch == "mmdit" else t64(tok)
    shift, scale = F.linear(F.silu(t64(c)), T["final.mod.w"], T["final.mod.b"]).chunk(2, dim=-1)
    y = F.linear(F.layer_norm(img, (sh.hidden,), eps=1e-6) * (1 + scale[:, None]) + shift[:, None],
                 T["final.lin.w"], T["final.lin.b"])
    B, p = y.shape[0], sh.patch
    gh, gw = sh.lat_h // p, sh.lat_w // p
    if sh.lat_f > 0:
        y = y.reshape(B, sh.lat_f, gh, gw, sh.out_ch, 1, p, p).permute(0, 4, 1, 5, 2, 6, 3, 7)
        return y.reshape(B, sh.out_ch, sh.lat_f, sh.lat_h, sh.lat_w).numpy()
    y = y.reshape(B, gh, gw, sh.out_ch, p, p).permute(0, 3, 1, 4, 2, 5)
    return y.reshape(B, sh.out_ch, sh.lat_h, sh.lat_w).numpy()


@pytest.mark.parametrize("kind", ["dit", "mmdit", "video"])
def test_final_layer_matches_torch_composition(kind):
    if kind == "dit":
        sh = small_dit()
    elif kind == "mmdit":
        sh = small_mmdit()
    else:
        sh = small_mmdit(lat_f=2, lat_h=4, lat_w=6, patch_t=1, rope_dims=3)
    W = weights64(sh, seed=11, scale=5.0)
    tok = rnd(sh.batch_model, sh.tokens, sh.hidden, scale=2.0) + 0.7
    c = rnd(sh.batch_model, sh.hidden, scale=3.0)
    out = model.final_layer(W, sh, tok, c)
    np.testing.assert_allclose(out, torch_final(W, sh, tok, c), rtol=1e-11, atol=1e-11)
    assert out.shape == (sh.batch_model, sh.out_ch) + sh.latent_dims[2:]
    # the layer normalises each token: an affine change of a token's values
    # (positive scale) moves the output only through LayerNorm's eps = 1e-6
    # (relative 1e-7 at these variances)
    tok2 = tok * 3.0 + 11.0
    if sh.arch == "mmdit":
        tok2[:, :sh.txt_tokens] = 1e6   # text rows never reach the head
    np.testing.assert_allclose(model.final_layer(W, sh, tok2, c), out, rtol=0, atol=2e-6 * np.abs(out).max())


def test_step_update_uses_the_first_in_ch_channels_of_the_head():
    """A learned-sigma head (2 * in_ch channels): DDIM on the guided first
    in_ch channels; whatever the other channels hold, the latent does not
    move with them, and with eps equal to the true noise every step lands on
    the data.  Guidance combines [cond ; uncond] before the channel slice."""
    sh = small_dit(in_ch=4, out_ch=8, lat_h=4, lat_w=4, batch=2)
    N = 50
    ab = sampler.ddim_alpha_bar()
    ts = sampler.ddim_timesteps(N)
    x0, eps = rnd(2, 4, 4, 4), rnd(2, 4, 4, 4)
    x = np.sqrt(ab[ts[0]]) * x0 + np.sqrt(1 - ab[ts[0]]) * eps
    s = sh.cfg_scale
    for i in range(N):
        garbage = rnd(4, 4, 4, 4, scale=1e3)
        # cond half = eps + d, uncond half = eps + d * (s / (s - 1)): guided = eps
        d = rnd(2, 4, 4, 4)
        head = np.concatenate([np.concatenate([eps + d, eps + d * s / (s - 1)]), garbage], axis=1)
        x = sampler.step_update(sh, x, head, N, i)
    np.testing.assert_allclose(x, x0, rtol=1e-8, atol=1e-8)


def test_step_update_euler_on_the_velocity_channels():
    sh = small_mmdit(in_ch=4, out_ch=4, lat_h=4, lat_w=4)
    x = rnd(1, 4, 4, 4)
    v = rnd(1, 4, 4, 4)
    N = 10
    got = sampler.step_update(sh, x, v, N, 3)
    np.testing.assert_allclose(got, x - v / N, rtol=1e-13, atol=1e-13)
    sh8 = small_mmdit(in_ch=4, out_ch=8, lat_h=4, lat_w=4)
    head = np.concatenate([v, rnd(1, 4, 4, 4, scale=1e3)], axis=1)
    np.testing.assert_allclose(sampler.step_update(sh8, x, head, N, 3), got, rtol=1e-13, atol=1e-13)

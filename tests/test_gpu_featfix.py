"""The whole cached sampling path through the C ABI against the oracle, plus
the paper's invariants checked bitwise on the GPU (Eq. 5's local reset,
Exact-only == FeatFix, Verify == no sites, all-refresh == vanilla) and
run-to-run determinism."""

import numpy as np
import pytest
import torch

import oracle
from oracle import schedule as osched
from paper_2607_27842_gb300 import featfix as ff, synthetic as syn

from .gpu_helpers import Case, rel_l2, tol_block, tol_latent

pytestmark = pytest.mark.gpu


def small_dit_bf16():
    sh = syn.reduced(syn.SHAPES["dit_xl2"], n_dual=3, hidden=256, heads=4, head_dim=64, mlp=1024, lat_h=16,
                     lat_w=16, batch=2, n_classes=10)
    ref = syn.refresh_every(10, 4)
    return syn.Workload(sh, 10, 2, ref, syn.diagonal_sites(10, 3, ref, 3))


def small_flux(dtype="bf16"):
    sh = syn.reduced(syn.SHAPES["flux"], n_dual=2, n_single=2, hidden=256, heads=2, head_dim=128, mlp=1024,
                     lat_h=16, lat_w=16, txt_tokens=12, dtype=dtype)
    ref = syn.refresh_every(8, 3)
    return syn.Workload(sh, 8, 1, ref, syn.diagonal_sites(8, 4, ref, 2))


def small_qwen():
    sh = syn.reduced(syn.SHAPES["qwen"], n_dual=3, hidden=256, heads=2, head_dim=128, mlp=1024, lat_h=16, lat_w=16,
                     txt_tokens=7)
    ref = syn.refresh_every(9, 3)
    return syn.Workload(sh, 9, 2, ref, syn.diagonal_sites(9, 3, ref, 3))


def small_hunyuan():
    sh = syn.reduced(syn.SHAPES["hunyuan"], n_dual=2, hidden=256, heads=2, head_dim=128, mlp=1024, lat_f=3,
                     lat_h=8, lat_w=12, txt_tokens=5)
    ref = syn.refresh_every(7, 3)
    return syn.Workload(sh, 7, 1, ref, syn.diagonal_sites(7, 2, ref, 2))


WORKLOADS = {
    "tiny": lambda: syn.workload("tiny"),
    "dit_bf16": small_dit_bf16,
    "flux_bf16": small_flux,
    "flux_f32": lambda: small_flux("f32"),
    "qwen_bf16": small_qwen,
    "hunyuan_bf16": small_hunyuan,
}


@pytest.fixture(params=list(WORKLOADS))
def case(request, cuda):
    c = Case(WORKLOADS[request.param]())
    yield c
    c.close()


@pytest.mark.parametrize("mode", ["featfix", "verify"])
def test_sample_matches_oracle(case, mode):
    """Free-running cached trajectory: final latent, the sites logged in
    order, accounting; every logged value against Eq. 4 on the GPU's own
    captured tensors."""
    case.schedule(mode)
    lat = case.sample(seed=1)
    logs, cnt = ff.featfix_get_log(case.ctx)
    x_ref, logs_ref, cnt_ref = case.oracle_run(mode, seed=1)
    err = rel_l2(lat.cpu().numpy(), x_ref)
    assert err < tol_latent(case.sh), err
    assert {k: cnt[k] for k in cnt_ref} == cnt_ref
    assert cnt["steps_done"] == case.wl.steps
    assert [(e["step"], e["layer"]) for e in logs] == [(e["step"], e["layer"]) for e in logs_ref]
    assert all(np.isfinite(e["rel_l1"]) and e["rel_l1"] > 0 for e in logs)
    bufs = case.capture_sites(mode)
    lat2 = case.sample(seed=1)
    logs2, _ = ff.featfix_get_log(case.ctx)
    case.check_logs_teacher_forced(bufs, logs2, mode)
    # with captures a site step's drafted blocks are chained one by one
    # instead of in one pass per run of blocks: the same value up to rounding
    assert [(e["step"], e["layer"]) for e in logs2] == [(e["step"], e["layer"]) for e in logs]
    assert rel_l2(lat2.cpu().numpy(), lat.cpu().numpy()) < (1e-5 if case.sh.dtype == "f32" else 1e-2)
    ff.featfix_debug_capture(case.ctx, -1, 0, None, None)


@pytest.mark.parametrize("mode", ["featfix", "verify"])
def test_site_history_push_matches_oracle(case, mode):
    """FEATFIX_FLAG_SITE_UPDATES_HISTORY: sites push their exact increment
    onto their block's history; trajectory, logs and accounting against the
    oracle run with the same reading."""
    flags = ff.FLAG_SITE_UPDATES_HISTORY
    case.schedule(mode, flags=flags)
    lat = case.sample(seed=1)
    logs, cnt = ff.featfix_get_log(case.ctx)
    x_ref, logs_ref, cnt_ref = case.oracle_run(mode, seed=1, site_updates_history=True)
    err = rel_l2(lat.cpu().numpy(), x_ref)
    assert err < tol_latent(case.sh), err
    assert {k: cnt[k] for k in cnt_ref} == cnt_ref
    assert [(e["step"], e["layer"]) for e in logs] == [(e["step"], e["layer"]) for e in logs_ref]
    bufs = case.capture_sites(mode, flags)
    case.sample(seed=1)
    case.check_logs_teacher_forced(bufs, ff.featfix_get_log(case.ctx)[0], mode, site_updates_history=True)
    ff.featfix_debug_capture(case.ctx, -1, 0, None, None)
    # the reading changes the trajectory when a site precedes a drafted step
    x_def, _, _ = case.oracle_run(mode, seed=1)
    assert np.abs(x_ref - x_def).max() > 0


@pytest.mark.parametrize("axis", ["tokens", "channels"])
def test_partial_forwarding_matches_oracle(case, axis):
    """Token / channel partial forwarding at FeatFix sites against the
    oracle; the all-selected mask is FeatFix bitwise and the none-selected
    mask is the per-block Verify trajectory bitwise."""
    n = case.sh.tokens if axis == "tokens" else case.sh.hidden
    ax = ff.MASK_TOKENS if axis == "tokens" else ff.MASK_CHANNELS
    mask = (np.arange(n) % 3 == 0).astype(np.uint8)
    case.schedule("featfix")
    ff.featfix_set_forward_mask(case.ctx, ax, mask)
    lat = case.sample(seed=1)
    x_ref, _, cnt_ref = case.oracle_run("featfix", seed=1, forward_mask=(axis, mask))
    err = rel_l2(lat.cpu().numpy(), x_ref)
    assert err < tol_latent(case.sh), err
    _, cnt = ff.featfix_get_log(case.ctx)
    assert {k: cnt[k] for k in cnt_ref} == cnt_ref
    ff.featfix_set_forward_mask(case.ctx, ax, np.ones(n, np.uint8))
    ones = case.sample(seed=1)
    ff.featfix_set_forward_mask(case.ctx, ff.MASK_NONE)
    whole = case.sample(seed=1)
    # per-block drafts in both arms (the default evaluates site-free drafted
    # steps in one telescoped pass, equal only up to rounding)
    case.schedule("featfix", flags=ff.FLAG_PER_BLOCK_DRAFT)
    ff.featfix_set_forward_mask(case.ctx, ax, np.zeros(n, np.uint8))
    zeros = case.sample(seed=1)
    ff.featfix_set_forward_mask(case.ctx, ff.MASK_NONE)
    case.schedule("verify", flags=ff.FLAG_PER_BLOCK_DRAFT)
    verify = case.sample(seed=1)
    assert torch.equal(ones, whole)
    assert torch.equal(zeros, verify)
    assert not torch.equal(lat, whole) and not torch.equal(lat, verify)
    with pytest.raises(ff.FeatFixError):
        ff.featfix_set_forward_mask(case.ctx, ax, np.ones(n + 1, np.uint8))


def test_blocks_teacher_forced(case):
    """Every block of the trajectory on the GPU's own incoming state: exact
    blocks vs B_l (Eq. 1), drafts vs Eq. 2 over the GPU's refresh increments."""
    wl, sh = case.wl, case.sh
    case.schedule("featfix")
    L = sh.n_layers
    kinds, keff, _ = ff.featfix_get_plan(case.ctx, wl.steps, L)
    picks = [(i, l) for i in range(wl.steps) for l in range(L)]
    if len(picks) > 30:
        picks = [p for p in picks if kinds[p] != ff.PLAN_DRAFT or p[1] % 3 == 0][:30]
    bufs = {}
    for (i, l) in picks:
        bufs[(i, l)] = (case.act_buffer(), case.act_buffer())
        ff.featfix_debug_capture(case.ctx, i, l, *bufs[(i, l)])
    # refresh increments of every layer for the draft checks
    inc = {}
    for i in wl.refresh:
        for l in range(L):
            if (i, l) not in bufs:
                bufs[(i, l)] = (case.act_buffer(), case.act_buffer())
                ff.featfix_debug_capture(case.ctx, i, l, *bufs[(i, l)])
    case.sample(seed=1)
    for i in wl.refresh:
        for l in range(L):
            u, h = bufs[(i, l)]
            inc[(i, l)] = case.to_logical(h) - case.to_logical(u)
    ang = oracle.model.rope_table(sh)
    for (i, l) in picks:
        u = case.to_logical(bufs[(i, l)][0])
        h = case.to_logical(bufs[(i, l)][1])
        k = kinds[i, l]
        if k == ff.PLAN_DRAFT:
            hist = [(s, inc[(s, l)]) for s in sorted([r for r in wl.refresh if r <= i], reverse=True)]
            ref = oracle.draft.draft(u, hist[:wl.K + 1], i, wl.K)
            tol = 1e-6 if sh.dtype == "f32" else 8e-3
        else:
            ref = oracle.featfix.block_at(case.W64, sh, l, i, wl.steps, u, case.cond64)
            tol = tol_block(sh)
        assert rel_l2(h, ref) < tol, (i, l, k, rel_l2(h, ref))
    ff.featfix_debug_capture(case.ctx, -1, 0, None, None)


def test_featfix_site_forwards_exact_output_bitwise(case):
    """Eq. 5: at a site the forwarded tensor is B_l(u) from the same u."""
    wl = case.wl
    case.schedule("featfix")
    i, l = wl.sites[0]
    u, h = case.act_buffer(), case.act_buffer()
    ff.featfix_debug_capture(case.ctx, i, l, u, h)
    case.sample(seed=3)
    hf = case.act_buffer()
    ff.featfix_debug_block(case.ctx, i, l, u, hf, case.cond)
    torch.cuda.synchronize()
    assert torch.equal(h, hf)


@pytest.mark.parametrize("flags", [0, ff.FLAG_PER_BLOCK_DRAFT], ids=["telescoped", "per_block"])
def test_arms_bitwise(case, flags):
    """Exact-only == FeatFix; Verify == schedule without sites; all-refresh ==
    vanilla; two runs identical -- with drafted steps evaluated in one pass
    and chained block by block."""
    wl = case.wl
    runs = {}
    for tag, mode, sites, refresh in (("featfix", "featfix", None, None), ("exact_only", "exact_only", None, None),
                                      ("verify", "verify", None, None), ("nosite", "featfix", (), None),
                                      ("allref", "featfix", (), tuple(range(wl.steps))),
                                      ("vanilla", "vanilla", None, None)):
        case.schedule(mode, refresh=refresh, sites=sites, flags=flags)
        runs[tag] = case.sample(seed=5).clone()
        runs[tag + "_log"] = ff.featfix_get_log(case.ctx)
    assert torch.equal(runs["featfix"], runs["exact_only"])
    assert torch.equal(runs["verify"], runs["nosite"])
    assert torch.equal(runs["allref"], runs["vanilla"])
    assert not torch.equal(runs["featfix"], runs["verify"])
    n = len(wl.sites)
    assert runs["featfix_log"][1]["forwarded"] == n and runs["verify_log"][1]["forwarded"] == 0
    assert runs["exact_only_log"][0] == [] and runs["exact_only_log"][1]["paid_checks"] == n
    assert runs["vanilla_log"][1]["refresh_steps"] == wl.steps
    # same state at the first paid check in both arms -> same logged value
    assert runs["featfix_log"][0][0]["rel_l1"] == runs["verify_log"][0][0]["rel_l1"]
    case.schedule("featfix", flags=flags)
    again = case.sample(seed=5)
    assert torch.equal(again, runs["featfix"])
    assert ff.featfix_get_log(case.ctx)[0] == runs["featfix_log"][0]


def test_telescoped_steps_match_per_block(case):
    """A drafted step evaluated in one pass over the refresh sums
    x_L - x_0 equals chaining the per-block drafts up to rounding."""
    case.schedule("featfix")
    a = case.sample(seed=7).cpu().numpy()
    case.schedule("featfix", flags=ff.FLAG_PER_BLOCK_DRAFT)
    b = case.sample(seed=7).cpu().numpy()
    assert rel_l2(a, b) < (1e-5 if case.sh.dtype == "f32" else 1e-2)


def test_fused_layernorm_matches_standalone(case):
    """Eq. 1's adaLN LayerNorm fused across the dense layers (FLAG_FUSED_LN,
    bf16: the producing GEMM writes x(1 + scale) and row statistics, the
    consuming GEMM corrects per row with (1 + scale)W^T and shift W^T) equals
    the standalone row kernel up to rounding; fp32 never fuses."""
    case.schedule("vanilla")
    a = case.sample(seed=11).cpu().numpy()
    case.schedule("vanilla", flags=ff.FLAG_FUSED_LN)
    b = case.sample(seed=11).cpu().numpy()
    if case.sh.dtype == "f32":
        np.testing.assert_array_equal(a, b)
    else:
        assert 0 < rel_l2(a, b) < 1e-2
    case.schedule("featfix")
    a = case.sample(seed=11).cpu().numpy()
    case.schedule("featfix", flags=ff.FLAG_FUSED_LN)
    b = case.sample(seed=11).cpu().numpy()
    assert rel_l2(a, b) < (1e-7 if case.sh.dtype == "f32" else 1e-2)
    x_ref, _, _ = case.oracle_run("featfix", seed=11)
    assert rel_l2(b, x_ref) < tol_latent(case.sh)


def test_call_order_errors(cuda):
    c = Case(syn.workload("tiny"))
    try:
        lat = torch.zeros(c.sh.latent_dims, device=cuda)
        with pytest.raises(ff.FeatFixError) as e:
            ff.featfix_step(c.ctx, lat, 0, c.cond)
        assert e.value.status == ff.ERR_STATE
        c.schedule("featfix")
        with pytest.raises(ff.FeatFixError) as e:
            ff.featfix_step(c.ctx, lat, 3, c.cond)
        assert e.value.status == ff.ERR_STATE
        with pytest.raises(ff.FeatFixError) as e:
            ff.featfix_sample(c.ctx, 1, 9, c.cond, lat)
        assert e.value.status == ff.ERR_SCHEDULE
        with pytest.raises(ff.FeatFixError) as e:
            ff.featfix_set_schedule(c.ctx, 10, (0, 3), 1, ((3, 1),))
        assert e.value.status == ff.ERR_SCHEDULE
        # step-wise driving equals featfix_sample
        c.schedule("featfix")
        ref = c.sample(seed=4)
        import oracle as orc
        x = torch.from_numpy(orc.noise.initial_latent(4, c.sh)).to(cuda)
        for i in range(c.wl.steps):
            ff.featfix_step(c.ctx, x, i, c.cond)
        torch.cuda.synchronize()
        assert rel_l2(x.cpu().numpy(), ref.cpu().numpy()) < 1e-6
    finally:
        c.close()


def test_sample_host_matches_device(cuda):
    c = Case(small_dit_bf16())
    try:
        c.schedule("featfix")
        ref = c.sample(seed=9).cpu()
        cond_h = c.cond_cpu.pin_memory()
        out_h = torch.empty(c.sh.latent_dims, dtype=torch.float32).pin_memory()
        ff.featfix_sample_host(c.ctx, 9, c.wl.steps, cond_h, out_h)
        assert torch.equal(out_h, ref)
    finally:
        c.close()

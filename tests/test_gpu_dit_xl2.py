"""The DiT-XL/2-shaped bf16 workload (28 blocks, hidden 1152, 16 heads x 72,
MLP 4608, 32x32x4 latent, patch 2, DDIM 50, order-2 draft, refresh every 5,
8 sites) at full size against the oracle."""

import numpy as np
import pytest
import torch

import oracle
from paper_2607_27842_gb300 import featfix as ff, synthetic as syn

from .gpu_helpers import Case, rel_l2

pytestmark = pytest.mark.gpu


def test_full_depth_trajectory_matches_oracle(cuda):
    """All 28 blocks and 50 steps free-running, one guided sample (model
    batch 2): final latent within 5e-2, every logged discrepancy close."""
    wl = syn.workload("dit_xl2")
    wl = syn.Workload(syn.reduced(wl.shape, batch=1), wl.steps, wl.K, wl.refresh, wl.sites)
    c = Case(wl)
    try:
        c.schedule("featfix")
        lat = c.sample(seed=1)
        logs, cnt = ff.featfix_get_log(c.ctx)
        x_ref, logs_ref, cnt_ref = c.oracle_run("featfix", seed=1)
        assert rel_l2(lat.cpu().numpy(), x_ref) < 5e-2
        assert {k: cnt[k] for k in cnt_ref} == cnt_ref == {"refresh_steps": 10, "paid_checks": 8, "forwarded": 8}
        assert [(g["step"], g["layer"]) for g in logs] == [(r["step"], r["layer"]) for r in logs_ref]
        bufs = c.capture_sites("featfix")
        c.sample(seed=1)
        c.check_logs_teacher_forced(bufs, ff.featfix_get_log(c.ctx)[0], "featfix")
    finally:
        c.close()


def test_bench_workload_blocks_teacher_forced(cuda):
    """The benchmarked configuration (batch 8 doubled to 16 by guidance):
    sampled exact blocks, one drafted block and one site, each on the GPU's
    own incoming state, within the per-block tolerance 2e-2; the site
    forwards B_l(u) bit for bit."""
    wl = syn.workload("dit_xl2")
    c = Case(wl, weights_on_gpu=True)
    try:
        c.schedule("featfix")
        site = wl.sites[0]
        picks = [(0, 0), (5, 27), site, (7, 13), (48, 20)]
        bufs = {p: (c.act_buffer(), c.act_buffer()) for p in picks}
        for r in (5, 0):
            bufs[(r, 13)] = (c.act_buffer(), c.act_buffer())
        for p, (u, h) in bufs.items():
            ff.featfix_debug_capture(c.ctx, p[0], p[1], u, h)
        c.sample(seed=1)
        hf = c.act_buffer()
        ff.featfix_debug_block(c.ctx, site[0], site[1], bufs[site][0], hf, c.cond)
        torch.cuda.synchronize()
        assert torch.equal(hf, bufs[site][1])
        L = wl.shape.n_layers
        kinds, keff, _ = ff.featfix_get_plan(c.ctx, wl.steps, L)
        names = [n for n, _ in ff.weight_spec(wl.shape) if not n.startswith("blk")]
        for (i, l) in [(0, 0), (5, 27), site, (48, 20)]:
            pre = "blk%d." % l
            W = c.W64_subset(names + [n for n, _ in ff.weight_spec(wl.shape) if n.startswith(pre)])
            u = c.to_logical(bufs[(i, l)][0])
            h = c.to_logical(bufs[(i, l)][1])
            ref = oracle.featfix.block_at(W, wl.shape, l, i, wl.steps, u, c.cond64)
            assert rel_l2(h, ref) < 2e-2, (i, l, rel_l2(h, ref))
        # drafted block (7, 13): order 1 at step 7 from refreshes 5 and 0
        assert kinds[7, 13] == ff.PLAN_DRAFT and keff[7] == 1
        inc = {r: c.to_logical(bufs[(r, 13)][1]) - c.to_logical(bufs[(r, 13)][0]) for r in (5, 0)}
        u = c.to_logical(bufs[(7, 13)][0])
        ref = oracle.draft.draft(u, [(5, inc[5]), (0, inc[0])], 7, wl.K)
        assert rel_l2(c.to_logical(bufs[(7, 13)][1]), ref) < 8e-3
        logs, cnt = ff.featfix_get_log(c.ctx)
        assert len(logs) == 8 and all(np.isfinite(e["rel_l2"]) and e["rel_l2"] > 0 for e in logs)
    finally:
        c.close()

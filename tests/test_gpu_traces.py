"""Mechanism traces (paper_2607_27842_gb300.traces) against the same traces
taken from the oracle's trajectories: the distance of the Verify and FeatFix
arms to the vanilla trajectory after a paid site, and the paid-layer sweep
of the final latent.  fp32 workloads, where the distances between arms are
far above the arithmetic's rounding."""

import numpy as np
import pytest

import oracle
from oracle import schedule as osched
from paper_2607_27842_gb300 import traces, synthetic as syn

from .gpu_helpers import Case
from .test_gpu_featfix import small_flux

pytestmark = pytest.mark.gpu


def oracle_rel_l1(a, ref):
    return float(np.abs(a - ref).sum() / np.abs(ref).sum())


def oracle_outputs(case, mode, points, sites=None):
    got = {}
    def hook(i, l, kind, u, h, extra):
        if (i, l) in points:
            got[(i, l)] = h.copy()
    x, _, _ = case.oracle_run(mode, seed=1, hook=hook, sites=sites)
    return got, x


def close(g, r):
    return abs(g - r) <= 0.02 * abs(r) + 1e-6


@pytest.mark.parametrize("make", [lambda: syn.workload("tiny"), lambda: small_flux("f32")], ids=["tiny", "flux_f32"])
def test_downstream_trace_matches_oracle(cuda, make):
    c = Case(make())
    try:
        rows = traces.downstream_trace(c.ctx, c.sh, c.wl, c.cond, seed=1)
        pts = {(r["step"], r["layer"]) for r in rows}
        ref = {m: oracle_outputs(c, m, pts)[0] for m in ("vanilla", "verify", "featfix")}
        for r in rows:
            p = (r["step"], r["layer"])
            ev = oracle_rel_l1(ref["verify"][p], ref["vanilla"][p])
            ef = oracle_rel_l1(ref["featfix"][p], ref["vanilla"][p])
            assert close(r["verify"], ev) and close(r["featfix"], ef), (r, ev, ef)
        # the arms coincide before the site and diverge from it on
        i0, l0 = sorted(c.wl.sites)[0]
        assert rows[0]["step"] == i0 and rows[0]["layer"] == l0
        assert any(abs(r["reduction"]) > 0 for r in rows)
    finally:
        c.close()


def test_paid_layer_sweep_matches_oracle(cuda):
    c = Case(syn.workload("tiny"))
    try:
        step = 4
        rows = traces.paid_layer_sweep(c.ctx, c.sh, c.wl, c.cond, step, layers=[0, 2, 3], seed=1)
        _, van = oracle_outputs(c, "vanilla", set())
        for r in rows:
            s = [(step, r["layer"])]
            _, v = oracle_outputs(c, "verify", set(), sites=s)
            _, f = oracle_outputs(c, "featfix", set(), sites=s)
            assert close(r["verify"], oracle_rel_l1(v, van)), r
            assert close(r["featfix"], oracle_rel_l1(f, van)), r
    finally:
        c.close()

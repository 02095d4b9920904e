"""The C ABI library without a GPU: it loads, exports every declared symbol,
and its host-only logic (schedule, draft weights, layout, argument checks)
agrees with the oracle."""

import ctypes
import os
import re

import numpy as np
import pytest

from oracle import draft as odraft, schedule as osched
from paper_2607_27842_gb300 import featfix as ff, synthetic as syn

from .conftest import ROOT, golden_lines


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(ff.LIB_PATH):
        from paper_2607_27842_gb300 import build
        build.build()
    return ff.lib()


def declared_symbols():
    names = set()
    for h in ("featfix.h", "featfix_ops.h"):
        src = open(os.path.join(ROOT, "include", h)).read()
        names |= set(re.findall(r"FEATFIX_API\s+[\w\s\*]+?\b(featfix_\w+)\s*\(", src))
    return names


def test_library_exports_every_declared_symbol(lib):
    names = declared_symbols()
    assert len(names) >= 20
    for n in names:
        assert hasattr(lib, n), n
    assert names == set(ff.SIGNATURES)


def test_status_strings(lib):
    for s in range(7):
        assert lib.featfix_status_string(s)
    assert lib.featfix_last_error(None) == b"null context"


@pytest.mark.parametrize("name", list(syn.SHAPES))
def test_weight_count_matches_spec(lib, name):
    sh = syn.SHAPES[name]
    assert ff.featfix_weight_count(sh) == len(ff.weight_spec(sh))


def test_invalid_descriptions_are_rejected(lib):
    sh = syn.SHAPES["tiny"]
    bad = [syn.reduced(sh, hidden=130), syn.reduced(sh, head_dim=36, heads=4, hidden=144),
           syn.reduced(sh, lat_h=7, patch=2), syn.reduced(sh, batch=0), syn.reduced(sh, rope_dims=2)]
    for b in bad:
        assert ff.featfix_weight_count(b) == -1
        d = ff.model_desc(b)
        out = ctypes.c_void_p()
        ptrs = (ctypes.c_void_p * 1)(16)
        assert lib.featfix_create(ctypes.byref(d), ptrs, 1, None, ctypes.byref(out)) == ff.ERR_INVALID_ARG
        assert out.value is None


def test_token_rows_are_text_first_stream_major(lib):
    sh = syn.reduced(syn.SHAPES["qwen"], lat_h=8, lat_w=8, txt_tokens=3)   # 16 image tokens, B_model 2
    rows = sorted(ff.featfix_token_row(sh, b, n) for b in range(2) for n in range(19))
    assert rows == list(range(38))
    assert ff.featfix_token_row(sh, 1, 2) == 5
    assert ff.featfix_token_row(sh, 0, 3) == 6
    assert ff.featfix_token_row(sh, 1, 3) == 6 + 16
    assert ff.featfix_token_row(sh, 2, 0) == -1


def test_plan_matches_hand_derivation(lib):
    wl = syn.workload("tiny")
    kinds, keff, w = ff.featfix_plan_build(wl.steps, 4, wl.refresh, wl.K, wl.sites)
    letters = "EDS"
    for line in golden_lines("plan_tiny.txt"):
        f = line.split()
        i = int(f[0])
        assert "".join(letters[k] for k in kinds[i]) == f[1]
        assert keff[i] == int(f[2])
        assert w[i, 0] == pytest.approx(float(f[3]), abs=1e-15)
        assert w[i, 1] == pytest.approx(float(f[4]), abs=1e-15)


def implied_weights(t, s, variant):
    """Oracle's Taylor forecast (Eq. 2) applied to unit increments."""
    out = []
    for j in range(len(s)):
        R = [np.array([1.0 if m == j else 0.0]) for m in range(len(s))]
        out.append(odraft.taylor_forecast(t, s, R, variant)[0])
    return out


@pytest.mark.parametrize("name", list(syn.SHAPES))
@pytest.mark.parametrize("mode", ["featfix", "verify", "exact_only", "vanilla"])
def test_plan_matches_oracle_on_every_workload(lib, name, mode):
    wl = syn.workload(name)
    L = wl.shape.n_layers
    kinds, keff, w = ff.featfix_plan_build(wl.steps, L, wl.refresh, wl.K, wl.sites, mode)
    okind, okeff = osched.build_plan(wl.steps, L, wl.refresh, wl.K, wl.sites, mode)
    np.testing.assert_array_equal(kinds, np.array(okind, dtype=np.uint8))   # bit-exact decisions
    hist = []
    for i in range(wl.steps):
        if i in wl.refresh:
            hist.insert(0, i)
            del hist[wl.K + 1:]
        drafted = mode != "vanilla" and i not in wl.refresh
        if not drafted:
            assert keff[i] == -1
            continue
        assert keff[i] == okeff[i]
        ref = implied_weights(i, hist[:okeff[i] + 1], "interp")
        np.testing.assert_allclose(w[i, :len(ref)], ref, rtol=1e-12, atol=1e-12)
        assert np.all(w[i, len(ref):] == 0)


def test_recursive_flag_matches_oracle_variant(lib):
    steps, refresh, K = 30, (0, 4, 9, 15, 22), 3
    _, keff, w = ff.featfix_plan_build(steps, 2, refresh, K, (), "featfix", ff.FLAG_TAYLOR_RECURSIVE)
    for i in (5, 12, 20, 29):
        s = sorted([r for r in refresh if r <= i], reverse=True)[:keff[i] + 1]
        ref = implied_weights(i, s, "recursive")
        np.testing.assert_allclose(w[i, :len(ref)], ref, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("name", list(syn.SHAPES))
@pytest.mark.parametrize("mode", ["featfix", "verify", "exact_only"])
@pytest.mark.parametrize("push", [False, True])
def test_block_plan_matches_oracle_histories(lib, name, mode, push):
    """Per-(step, block) draft weights against the oracle's per-block history
    steps, with and without sites pushing their increments."""
    wl = syn.workload(name)
    L = wl.shape.n_layers
    flags = ff.FLAG_SITE_UPDATES_HISTORY if push else 0
    keff, w = ff.featfix_plan_build_blocks(wl.steps, L, wl.refresh, wl.K, wl.sites, mode, flags)
    _, keff_step, w_step = ff.featfix_plan_build(wl.steps, L, wl.refresh, wl.K, wl.sites, mode, flags)
    hs = osched.block_history_steps(wl.steps, L, wl.refresh, wl.K, wl.sites, mode, push)
    site_set = {tuple(x) for x in wl.sites}
    for i in range(wl.steps):
        for l in range(L):
            if hs[i][l] is None:
                assert keff[i, l] == -1
                continue
            assert keff[i, l] == len(hs[i][l]) - 1 == min(wl.K, len(hs[i][l]) - 1)
            ref = implied_weights(i, hs[i][l], "interp")
            np.testing.assert_allclose(w[i, l, :len(ref)], ref, rtol=1e-12, atol=1e-12)
            if not push:   # without pushes every block reads the refresh-only history
                assert keff[i, l] == keff_step[i]
                np.testing.assert_array_equal(w[i, l], w_step[i])
    if push and wl.sites:
        # a block whose site precedes a drafted step reads that site step
        i0, l0 = sorted(site_set)[0]
        later = [i for i in range(i0 + 1, wl.steps) if i not in wl.refresh]
        if later and later[0] < min([r for r in wl.refresh if r > i0], default=wl.steps):
            assert hs[later[0]][l0][0] == i0


@pytest.mark.parametrize("bad,status", [
    (dict(refresh=(1, 3)), ff.ERR_SCHEDULE),
    (dict(sites=((3, 0),)), ff.ERR_SCHEDULE),
    (dict(sites=((4, 9),)), ff.ERR_SCHEDULE),
    (dict(sites=((4, 1), (4, 1))), ff.ERR_SCHEDULE),
    (dict(K=4), ff.ERR_SCHEDULE),
    (dict(refresh=(0, 0, 3)), ff.ERR_SCHEDULE),
    (dict(refresh=(0, 10)), ff.ERR_SCHEDULE),
    (dict(mode=7), ff.ERR_INVALID_ARG),
])
def test_plan_rules_give_status_codes(lib, bad, status):
    args = dict(refresh=(0, 3, 6, 9), K=1, sites=((4, 2),), mode="featfix")
    args.update(bad)
    with pytest.raises(ff.FeatFixError) as ei:
        ff.featfix_plan_build(10, 4, args["refresh"], args["K"], args["sites"], args["mode"])
    assert ei.value.status == status


def test_null_context_calls_fail_cleanly(lib):
    assert lib.featfix_step(None, None, 0, None) == ff.ERR_INVALID_ARG
    assert lib.featfix_get_log(None, None, 0, None, None) == ff.ERR_INVALID_ARG
    assert lib.featfix_set_schedule(None, 1, None, 0, 0, None, 0, 0, 0) == ff.ERR_INVALID_ARG
    lib.featfix_destroy(None)

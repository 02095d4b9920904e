"""Whole cached trajectories at full depth and width against stored oracle
runs (tests/golden/oracle_<workload>_<mode>.npz, written by
tests/golden/make_oracle_latents.py from the float64 oracle alone):

* dit_xl2     the benchmarked DiT-XL/2 configuration: 28 blocks, batch 8
              doubled to 16 by guidance, 50 DDIM steps, order-2 draft, 8 sites;
              FeatFix and Verify arms (Verify's paid checks run on a shadow
              copy of the step's input, the site-free drafted steps in one
              telescoped pass);
* flux_512    FLUX: 19 dual + 38 single blocks at width 3072, 512^2 image
              (1024 image + 512 text tokens), order-1 draft, 12 sites;
* qwen_512    Qwen-Image: 60 dual blocks at width 3072, 512^2 image
              (1024 image + 256 text tokens), guidance batch 2, order 2, 16 sites;
* hunyuan_3f  HunyuanVideo: 54 dual blocks at width 2048, 3-D rotary, 3 of the
              9 latent frames (4770 video + 256 text tokens), order 1, 12 sites.

The reduced token counts are the sizes at which a float64 oracle trajectory
finishes in hours on the host; depth, width, heads, schedule and sites are
the full workloads'.  Checked per trajectory (Section 3.3, Eqs. 2-5): the
final latent within 5e-2 relative L2 (bf16), the paid checks in the same
order, the accounting bit-exact, and every logged discrepancy against Eq. 4
evaluated by the oracle on the GPU's own captured tensors (2e-2).  The
FeatFix arm runs again with every drafted step chained block by block, and
with the adaLN LayerNorm fused across the dense layers.
"""

import importlib.util
import os

import numpy as np
import pytest
import torch

from paper_2607_27842_gb300 import featfix as ff, synthetic as syn

from .gpu_helpers import Case, rel_l2, tol_latent

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


def golden_module():
    spec = importlib.util.spec_from_file_location("make_oracle_latents",
                                                  os.path.join(HERE, "golden", "make_oracle_latents.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


GOLDEN = [("dit_xl2", "featfix"), ("dit_xl2", "verify"), ("flux_512", "featfix"), ("qwen_512", "featfix"),
          ("hunyuan_3f", "featfix")]


@pytest.mark.parametrize("name,mode", GOLDEN, ids=["%s-%s" % g for g in GOLDEN])
def test_trajectory_matches_stored_oracle(cuda, name, mode):
    gm = golden_module()
    stored = gm.load(name, mode)
    if stored is None:
        pytest.skip("no stored oracle run %s yet" % os.path.basename(gm.golden_path(name, mode)))
    x_ref, logs_ref, cnt_ref, meta = stored
    wl = syn.workload(name)
    # the stored run belongs to this oracle, these inputs and this schedule
    assert meta["digest"] == gm.code_digest(), "oracle changed since the stored run"
    assert meta["inputs"] == gm.input_fingerprint(wl), "seeded inputs changed since the stored run"
    want = gm.key(wl, mode)
    assert {k: meta[k] for k in want} == want
    c = Case(wl, seed=gm.SEED_WEIGHTS, keep_host=False)
    try:
        c.schedule(mode)
        lat = c.sample(seed=gm.SEED_LATENT)
        logs, cnt = ff.featfix_get_log(c.ctx)
        err = rel_l2(lat.cpu().numpy(), x_ref)
        assert err < tol_latent(c.sh), err
        assert {k: cnt[k] for k in cnt_ref} == cnt_ref
        assert [(e["step"], e["layer"]) for e in logs] == [(e["step"], e["layer"]) for e in logs_ref]
        assert all(np.isfinite(e["rel_l1"]) and e["rel_l1"] > 0 for e in logs)
        # logged values: teacher-forced on the GPU's own tensors at every site
        bufs = c.capture_sites(mode)
        lat2 = c.sample(seed=gm.SEED_LATENT)
        c.check_logs_teacher_forced(bufs, ff.featfix_get_log(c.ctx)[0], mode)
        assert rel_l2(lat2.cpu().numpy(), x_ref) < tol_latent(c.sh)
        del bufs
        ff.featfix_debug_capture(c.ctx, -1, 0, None, None)
        if mode == "featfix":
            # every drafted step chained block by block instead of one pass
            c.schedule(mode, flags=ff.FLAG_PER_BLOCK_DRAFT)
            lat3 = c.sample(seed=gm.SEED_LATENT)
            assert rel_l2(lat3.cpu().numpy(), x_ref) < tol_latent(c.sh)
            assert not torch.equal(lat3, lat)
            # the adaLN LayerNorm fused across the dense layers (opt-in)
            c.schedule(mode, flags=ff.FLAG_FUSED_LN)
            lat4 = c.sample(seed=gm.SEED_LATENT)
            assert rel_l2(lat4.cpu().numpy(), x_ref) < tol_latent(c.sh)
    finally:
        c.close()

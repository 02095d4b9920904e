"""Mechanism traces of the cached sampler on random weights (the paper's
feature-trace study, Section 3.2 and the downstream / paid-layer analyses of
Section 4): how far the Verify and FeatFix trajectories sit from the vanilla
(all-exact) trajectory, block by block after a paid site, and at the final
latent when the site's layer is varied.

Everything runs through the C ABI (featfix_sample with debug captures of the
forwarded block outputs); only the relative-L1 distances between captured
tensors are taken here, with PyTorch reductions on the GPU -- an analysis of
the path's outputs, not part of it.
"""

import torch

from . import featfix as ff
from . import synthetic as syn


def rel_l1(a, ref):
    """||a - ref||_1 / ||ref||_1 (Eq. 4's measure, here against vanilla)."""
    a, ref = a.double(), ref.double()
    return float((a - ref).abs().sum() / ref.abs().sum().clamp_min(1e-30))


def _outputs(ctx, sh, wl, cond, seed, mode, points, sites=None, flags=0):
    """Forwarded block outputs at (step, layer) points and the final latent."""
    dt = syn.torch_dtype(sh)
    dev = cond.device
    ff.featfix_debug_capture(ctx, -1, 0, None, None)
    bufs = {}
    for (i, l) in points:
        bufs[(i, l)] = torch.empty((sh.batch_model * sh.tokens, sh.hidden), dtype=dt, device=dev)
        ff.featfix_debug_capture(ctx, i, l, None, bufs[(i, l)])
    ff.featfix_set_schedule(ctx, wl.steps, wl.refresh, wl.K, wl.sites if sites is None else sites, mode, flags)
    lat = torch.empty(sh.latent_dims, dtype=torch.float32, device=dev)
    ff.featfix_sample(ctx, seed, wl.steps, cond, lat)
    torch.cuda.synchronize(dev)
    ff.featfix_debug_capture(ctx, -1, 0, None, None)
    return bufs, lat


def downstream_trace(ctx, sh, wl, cond, seed=1, site=None, steps_after=1):
    """Relative-L1 distance to the vanilla trajectory of the Verify and the
    FeatFix arms at every block from the site's layer to the last, at the
    site's step and the next ``steps_after`` steps (a site of the schedule,
    the first one by default).  Rows: dict(step, layer, verify, featfix,
    reduction = verify - featfix)."""
    i0, l0 = site if site is not None else sorted(tuple(s) for s in wl.sites)[0]
    L = sh.n_layers
    points = [(i, l) for i in range(i0, min(wl.steps, i0 + steps_after + 1))
              for l in range(l0 if i == i0 else 0, L)]
    out = {}
    for mode in ("vanilla", "verify", "featfix"):
        b, _ = _outputs(ctx, sh, wl, cond, seed, mode, points)
        out[mode] = b
    rows = []
    for p in points:
        ev = rel_l1(out["verify"][p], out["vanilla"][p])
        ef = rel_l1(out["featfix"][p], out["vanilla"][p])
        rows.append({"step": p[0], "layer": p[1], "verify": ev, "featfix": ef, "reduction": ev - ef})
    return rows


def paid_layer_sweep(ctx, sh, wl, cond, step, layers, seed=1):
    """One paid site at (step, l) for each l: relative-L1 distance of the
    final latent to the vanilla latent under Verify and FeatFix.  Rows:
    dict(layer, verify, featfix, reduction)."""
    _, van = _outputs(ctx, sh, wl, cond, seed, "vanilla", [])
    rows = []
    for l in layers:
        s = [(step, l)]
        _, v = _outputs(ctx, sh, wl, cond, seed, "verify", [], sites=s)
        _, f = _outputs(ctx, sh, wl, cond, seed, "featfix", [], sites=s)
        ev, ef = rel_l1(v, van), rel_l1(f, van)
        rows.append({"layer": l, "verify": ev, "featfix": ef, "reduction": ev - ef})
    return rows

"""The FeatFix cached sampling loop, float64 (Section 3, Eqs. 1-5).

Per denoising step i the L blocks run in order on the incoming state u:

* EXACT (full refresh): h = B_l(u) (Eq. 1); the increment h - u is pushed
  onto block l's refresh history (newest first, K + 1 kept).
* DRAFT: h = D(u), the base policy's draft (Eq. 2, ``oracle.draft``).
* SITE (a paid check): the same-input pair h_d = D(u), h_f = B_l(u) (Eq. 3);
  the discrepancy ||h_d - h_f||_1 / (||h_f||_1 + eps) (Eq. 4) and its L2
  analogue are logged and never route the sample; the forwarded output is
  h_f for FeatFix (Eq. 5) and h_d for Verify.  Exact-only drops the draft and
  the discrepancy and forwards h_f.  By default a site's exact output does
  not enter the refresh history, so the draft policy outside S is the base
  policy's; with ``site_updates_history`` (the alternative reading of where
  the paper's differences are estimated) the site's increment h_f - u is
  pushed onto block l's history like a refresh, after its own draft.
* Vanilla: every block exact, no history.

Accounting (Section 3.3): full-refresh steps, paid checks and forwarded
corrections are counted separately.

Test infrastructure only.
"""

import numpy as np

from . import draft as _draft
from . import model as _model
from . import sampler as _sampler
from .schedule import EXACT, DRAFT, SITE, build_plan

EPS = 1e-8


def rel_l1(hd, hf):
    """Eq. 4."""
    return float(np.abs(hd - hf).sum() / (np.abs(hf).sum() + EPS))


def rel_l2(hd, hf):
    """The L2 analogue of Eq. 4 (the logged scalar of a metric ablation)."""
    return float(np.sqrt(((hd - hf) ** 2).sum()) / (np.sqrt((hf ** 2).sum()) + EPS))


def n_layers(shape):
    return shape.n_dual + shape.n_single if shape.arch == "mmdit" else shape.n_dual


def model_input(shape, x):
    """The model batch: the latent, duplicated for [cond ; uncond] under CFG."""
    return np.concatenate([x, x], axis=0) if shape.cfg else x


def forward_partial(hd, hf, mask):
    """Token- or channel-level partial forwarding arm (Section 3.2's
    alternatives to whole-block forwarding): the exact output on the
    selected tokens (axis 'tokens', mask over a sample's sequence) or
    channels (axis 'channels'), the draft elsewhere."""
    axis, m = mask
    m = np.asarray(m, dtype=bool)
    sel = m[None, :, None] if axis == "tokens" else m[None, None, :]
    return np.where(sel, hf, hd)


def run(W, shape, cond, x_T, steps, refresh, K, sites, mode="featfix",
        variant="interp", hook=None, site_updates_history=False, forward_mask=None):
    """Run the cached sampler.

    W      dict of float64 weights.
    cond   DiT: int labels [B_model]; MMDiT: text tokens [B_model, N_txt, C].
    x_T    initial latent [B_lat, ...].
    sites  (step, layer) pairs.
    hook   optional callable(step, layer, kind, u, h_out, extra) for tests.
    site_updates_history   push a site's exact increment onto its block's
           history (after the site's own draft).
    forward_mask  None (whole-block forwarding) or ('tokens', mask[N_tot]) /
           ('channels', mask[C]): the FeatFix arm forwards h_f only there.

    Returns (x_0, logs, counters) with logs = list of dicts
    {step, layer, rel_l1, rel_l2} in execution order and counters =
    {refresh_steps, paid_checks, forwarded}.
    """
    L = n_layers(shape)
    kind, _ = build_plan(steps, L, refresh, K, sites, mode)
    rs = set(refresh)
    ang = _model.rope_table(shape)
    hist = [[] for _ in range(L)]
    logs = []
    counters = {"refresh_steps": 0, "paid_checks": 0, "forwarded": 0}
    x = np.asarray(x_T, dtype=np.float64)
    bm = shape.batch * (2 if shape.cfg else 1)
    for i in range(steps):
        t = _sampler.model_time(shape.sampler, steps, i)
        if mode == "vanilla" or i in rs:
            counters["refresh_steps"] += 1
        labels = cond if shape.arch == "dit" else None
        c = _model.cond_vector(W, t, labels=labels, batch=bm)
        tok = _model.embed_tokens(W, shape, model_input(shape, x),
                                  txt=None if shape.arch == "dit" else cond)
        for l in range(L):
            u = tok
            k = kind[i][l]
            extra = None
            if k == EXACT:
                h = _model.exact_block(W, shape, l, u, c, ang)
                if mode != "vanilla":
                    hist[l].insert(0, (i, h - u))
                    del hist[l][K + 1:]
            elif k == DRAFT:
                h = _draft.draft(u, hist[l], i, K, variant)
            else:
                counters["paid_checks"] += 1
                hf = _model.exact_block(W, shape, l, u, c, ang)
                if mode == "exact_only":
                    h = hf
                    counters["forwarded"] += 1
                else:
                    hd = _draft.draft(u, hist[l], i, K, variant)
                    logs.append({"step": i, "layer": l, "rel_l1": rel_l1(hd, hf), "rel_l2": rel_l2(hd, hf)})
                    if mode == "featfix":
                        h = hf if forward_mask is None else forward_partial(hd, hf, forward_mask)
                        counters["forwarded"] += 1
                    else:
                        h = hd
                    extra = {"h_d": hd, "h_f": hf}
                if site_updates_history:
                    hist[l].insert(0, (i, hf - u))
                    del hist[l][K + 1:]
            if hook is not None:
                hook(i, l, k, u, h, extra)
            tok = h
        out = _model.final_layer(W, shape, tok, c)
        x = _sampler.step_update(shape, x, out, steps, i)
    return x, logs, counters


def block_at(W, shape, layer, step, steps, u, cond):
    """B_l(u; t_step, c) on a given incoming state (teacher-forced check)."""
    t = _sampler.model_time(shape.sampler, steps, step)
    bm = shape.batch * (2 if shape.cfg else 1)
    c = _model.cond_vector(W, t, labels=cond if shape.arch == "dit" else None, batch=bm)
    return _model.exact_block(W, shape, layer, np.asarray(u, dtype=np.float64), c)

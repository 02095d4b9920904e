"""Writes the stored oracle trajectories the full-size GPU parity tests compare
against: the final latent, the logged discrepancies of every paid check
(Eq. 4 and its L2 analogue) and the accounting of Section 3.3, from a whole
float64 oracle run of a workload's cached sampler.

Calls only ``oracle/`` for the arithmetic; ``synthetic`` supplies the seeded
inputs (the same weights, conditioning and initial latent the GPU tests
feed the CUDA path).  One file per (workload, mode):
``tests/golden/oracle_<workload>_<mode>.npz``, keyed by the workload, the
seeds, the schedule, the model dtype, a digest of the oracle's code (comments
and docstrings excluded) and a fingerprint of the seeded inputs, which the
tests check before comparing.

    OPENBLAS_NUM_THREADS=2 python tests/golden/make_oracle_latents.py dit_xl2:featfix
    OPENBLAS_NUM_THREADS=2 python tests/golden/make_oracle_latents.py hunyuan_3f:featfix   (and so on)

Much of an oracle block is single-threaded numpy, so several workloads run
side by side with a few BLAS threads each.  On eight x86 cores a DiT-XL/2
trajectory takes about an hour, the reduced-token MMDiT workloads a few
hours each (many hours at the full token counts).
"""

import argparse
import ast
import hashlib
import json
import os
import platform
import sys
import time

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

SEED_WEIGHTS, SEED_COND, SEED_LATENT = 0, 2, 1


def _strip_docstrings(tree):
    for node in ast.walk(tree):
        if isinstance(node, (ast.Module, ast.FunctionDef, ast.ClassDef, ast.AsyncFunctionDef)):
            body = node.body
            if body and isinstance(body[0], ast.Expr) and isinstance(getattr(body[0], "value", None), ast.Constant) \
                    and isinstance(body[0].value.value, str):
                node.body = body[1:] or [ast.Pass()]
    return tree


def code_digest():
    """sha256 over the syntax trees of oracle/*.py, so edits to comments or
    docstrings keep stored trajectories valid."""
    files = sorted(os.path.join(ROOT, "oracle", f) for f in os.listdir(os.path.join(ROOT, "oracle"))
                   if f.endswith(".py"))
    h = hashlib.sha256()
    for f in files:
        with open(f) as fh:
            tree = _strip_docstrings(ast.parse(fh.read()))
        h.update(os.path.basename(f).encode())
        h.update(ast.dump(tree).encode())
    return h.hexdigest()[:20]


def input_fingerprint(wl):
    """sha256 over a sample of the seeded inputs -- the first and last weight
    tensors, the conditioning and the initial latent -- so a stored trajectory
    is known to belong to the inputs the generator makes today."""
    import numpy as np
    import oracle
    from paper_2607_27842_gb300 import featfix, synthetic as syn
    sh = wl.shape
    names = [n for n, _ in featfix.weight_spec(sh)]
    pick = names[:3] + names[-2:]
    w = syn.make_weights(sh, seed=SEED_WEIGHTS, names=pick)
    h = hashlib.sha256()
    for n in pick:
        h.update(n.encode())
        h.update(syn.to_numpy64(w[n]).tobytes())
    h.update(np.ascontiguousarray(syn.oracle_cond(sh, syn.make_cond(sh, seed=SEED_COND)), dtype=np.float64).tobytes())
    h.update(np.ascontiguousarray(oracle.noise.initial_latent(SEED_LATENT, sh), dtype=np.float64).tobytes())
    return h.hexdigest()[:20]


def golden_path(workload, mode):
    return os.path.join(HERE, "oracle_%s_%s.npz" % (workload, mode))


def key(wl, mode):
    """What a stored trajectory depends on, besides the code digest."""
    import dataclasses
    return {"workload": wl.shape.name, "mode": mode, "shape": dataclasses.asdict(wl.shape), "steps": wl.steps,
            "K": wl.K, "refresh": list(wl.refresh), "sites": [list(s) for s in wl.sites],
            "seeds": {"weights": SEED_WEIGHTS, "cond": SEED_COND, "latent": SEED_LATENT}}


def load(workload, mode):
    """(final latent, logs, counters, meta) of a stored trajectory, or None."""
    import numpy as np
    p = golden_path(workload, mode)
    if not os.path.exists(p):
        return None
    z = np.load(p)
    meta = json.loads(str(z["meta"]))
    logs = [{"step": int(s), "layer": int(l), "rel_l1": float(a), "rel_l2": float(b)}
            for s, l, a, b in zip(z["site_step"], z["site_layer"], z["rel_l1"], z["rel_l2"])]
    counters = dict(zip(meta["counter_names"], [int(v) for v in z["counters"]]))
    return z["latent"].astype(np.float64), logs, counters, meta


def run(workload, mode, cache_gb):
    import numpy as np
    import oracle
    from paper_2607_27842_gb300 import synthetic as syn
    wl = syn.workload(workload)
    sh = wl.shape
    digest, inputs = code_digest(), input_fingerprint(wl)   # taken before the run: the code it ran
    W = syn.LazyOracleWeights(sh, seed=SEED_WEIGHTS, cache_bytes=int(cache_gb * 2 ** 30))
    cond = syn.oracle_cond(sh, syn.make_cond(sh, seed=SEED_COND))
    x_T = oracle.noise.initial_latent(SEED_LATENT, sh)
    t0 = time.time()
    last = [t0]

    def progress(step, layer, kind, u, h, extra):
        if layer == sh.n_layers - 1:
            now = time.time()
            print("%s/%s step %d done, %.1f s (total %.1f min)" % (workload, mode, step, now - last[0],
                                                                 (now - t0) / 60), flush=True)
            last[0] = now

    x, logs, counters = oracle.featfix.run(W, sh, cond, x_T, wl.steps, wl.refresh, wl.K, wl.sites, mode,
                                           hook=progress)
    elapsed = time.time() - t0
    names = sorted(counters)
    meta = dict(key(wl, mode), digest=digest, inputs=inputs, counter_names=names, elapsed_s=elapsed,
                host="%s, %d cores" % (platform.machine(), os.cpu_count() or 0),
                blas_threads=os.environ.get("OPENBLAS_NUM_THREADS", "default"))
    np.savez_compressed(golden_path(workload, mode), latent=x.astype(np.float32),
                        site_step=np.array([e["step"] for e in logs], dtype=np.int32),
                        site_layer=np.array([e["layer"] for e in logs], dtype=np.int32),
                        rel_l1=np.array([e["rel_l1"] for e in logs]), rel_l2=np.array([e["rel_l2"] for e in logs]),
                        counters=np.array([counters[k] for k in names], dtype=np.int64), meta=json.dumps(meta))
    print("wrote %s (%.1f min)" % (golden_path(workload, mode), elapsed / 60), flush=True)


def main():
    p = argparse.ArgumentParser()
    p.add_argument("jobs", nargs="+", help="workload:mode, e.g. dit_xl2:featfix")
    p.add_argument("--cache-gb", type=float, default=16.0,
                   help="host memory for model-dtype copies of block weights (the rest is regenerated)")
    p.add_argument("--skip-current", action="store_true", help="skip jobs whose stored file has the current digest")
    a = p.parse_args()
    for job in a.jobs:
        wname, mode = job.split(":")
        if a.skip_current:
            got = load(wname, mode)
            if got is not None and got[3].get("digest") == code_digest() \
                    and got[3].get("inputs") == input_fingerprint(__import__(
                        "paper_2607_27842_gb300.synthetic", fromlist=["workload"]).workload(wname)):
                print("current: %s" % job, flush=True)
                continue
        run(wname, mode, a.cache_gb)


if __name__ == "__main__":
    main()

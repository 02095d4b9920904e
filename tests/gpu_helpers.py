"""Shared helpers of the GPU parity tests (CUDA path vs the CPU oracle)."""

import numpy as np
import torch

import oracle
from paper_2607_27842_gb300 import featfix as ff, synthetic as syn


def rel_l2(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / (np.linalg.norm(b) + 1e-30))


def tol_block(shape):
    """Per-block output tolerance: 1e-4 in fp32 mode, 2e-2 in bf16 mode."""
    return 1e-4 if shape.dtype == "f32" else 2e-2


def tol_latent(shape):
    """Final-latent tolerance: 1e-4 in fp32 mode, 5e-2 in bf16 mode."""
    return 1e-4 if shape.dtype == "f32" else 5e-2


def tol_log(shape):
    """Logged discrepancy (Eq. 4 and its L2 analogue) against the oracle's
    evaluated on the GPU's own tensors: 1e-4 relative in fp32 mode, 2e-2 in
    bf16 mode.  Both sides then start from the same stored values (incoming
    state u, the history increments the draft reads, the exact output h^f),
    so only fp32 against fp64 arithmetic separates them."""
    return 1e-4 if shape.dtype == "f32" else 2e-2


class Case:
    """One model + schedule on cuda:0 with the matching oracle inputs."""

    def __init__(self, wl, seed=0, weights_on_gpu=False, keep_host=True):
        """weights_on_gpu: drawn by the GPU generator (other values than the
        oracle's CPU generator; for tests that compare on captured tensors).
        keep_host=False: CPU-generated values moved to the GPU tensor by
        tensor, with no host copy kept (the large models)."""
        self.wl = wl
        self.sh = sh = wl.shape
        self.dev = torch.device("cuda:0")
        if weights_on_gpu:
            self.w = syn.make_weights(sh, seed=seed, device=self.dev)
            self._w_cpu = None
        elif not keep_host:
            self.w = syn.make_weights(sh, seed=seed, to=self.dev)
            self._w_cpu = None
        else:
            self._w_cpu = syn.make_weights(sh, seed=seed)
            self.w = {k: v.to(self.dev) for k, v in self._w_cpu.items()}
        self.cond_cpu = syn.make_cond(sh, seed=2)
        self.cond = self.cond_cpu.to(self.dev)
        self.ctx = ff.featfix_create(sh, self.w)
        self._W64 = None

    @property
    def W64(self):
        if self._W64 is None:
            src = self._w_cpu if self._w_cpu is not None else {k: v.cpu() for k, v in self.w.items()}
            self._W64 = syn.oracle_weights(src)
        return self._W64

    def W64_subset(self, names):
        return {k: syn.to_numpy64(self.w[k]) for k in names}

    @property
    def cond64(self):
        return syn.oracle_cond(self.sh, self.cond_cpu)

    def schedule(self, mode="featfix", refresh=None, sites=None, flags=0):
        wl = self.wl
        ff.featfix_set_schedule(self.ctx, wl.steps, wl.refresh if refresh is None else refresh, wl.K,
                                wl.sites if sites is None else sites, mode, flags)

    def sample(self, seed=1):
        lat = torch.empty(self.sh.latent_dims, dtype=torch.float32, device=self.dev)
        ff.featfix_sample(self.ctx, seed, self.wl.steps, self.cond, lat)
        torch.cuda.synchronize()
        return lat

    def act_buffer(self):
        return torch.empty((self.sh.batch_model * self.sh.tokens, self.sh.hidden), dtype=syn.torch_dtype(self.sh),
                           device=self.dev)

    def rows(self):
        """Library row of every (sample, token), logical order."""
        sh = self.sh
        return np.array([[ff.featfix_token_row(sh, b, n) for n in range(sh.tokens)] for b in range(sh.batch_model)])

    def to_logical(self, buf):
        a = syn.to_numpy64(buf)
        return a[self.rows()]

    def from_logical(self, arr):
        sh = self.sh
        out = np.empty((sh.batch_model * sh.tokens, sh.hidden))
        out[self.rows().reshape(-1)] = np.asarray(arr).reshape(-1, sh.hidden)
        return torch.from_numpy(out).to(syn.torch_dtype(sh)).to(self.dev)

    def oracle_run(self, mode="featfix", seed=1, refresh=None, sites=None, hook=None, site_updates_history=False,
                   forward_mask=None):
        wl = self.wl
        return oracle.featfix.run(self.W64, self.sh, self.cond64, oracle.noise.initial_latent(seed, self.sh),
                                  wl.steps, wl.refresh if refresh is None else refresh, wl.K,
                                  wl.sites if sites is None else sites, mode, hook=hook,
                                  site_updates_history=site_updates_history, forward_mask=forward_mask)

    def capture_sites(self, mode="featfix", flags=0):
        """Register captures at every paid check of the schedule: the
        incoming state, the forwarded output and the history increments the
        site's draft reads.  Returns {(step, layer): (u, out, [hist...])}."""
        wl, sh = self.wl, self.sh
        keff, _ = ff.featfix_plan_build_blocks(wl.steps, sh.n_layers, wl.refresh, wl.K, wl.sites, mode, flags)
        bufs = {}
        for (i, l) in wl.sites:
            hist = [self.act_buffer() for _ in range(int(keff[i, l]) + 1)]
            u, out = self.act_buffer(), self.act_buffer()
            ff.featfix_debug_capture(self.ctx, i, l, u, out)
            ff.featfix_debug_capture_history(self.ctx, i, l, hist)
            bufs[(i, l)] = (u, out, hist)
        return bufs

    def check_logs_teacher_forced(self, bufs, logs, mode="featfix", site_updates_history=False):
        """Every logged discrepancy against Eq. 4 (and its L2 analogue)
        evaluated by the oracle on the GPU's own captured tensors: the draft
        h^d formed by the oracle's Taylor series (Eq. 2) from the captured
        history increments and rounded to the model dtype (the block output
        as it would be forwarded), h^f the forwarded output (FeatFix) or the exact
        block recomputed from the captured u (Verify; the GPU path is
        deterministic, so this is the h^f the check used)."""
        wl, sh = self.wl, self.sh
        got = {(e["step"], e["layer"]): e for e in logs}
        assert sorted(got) == sorted(bufs)
        tol = tol_log(sh)
        worst = 0.0
        for (i, l), (u, out, hist) in bufs.items():
            if mode == "featfix":
                hf_dev = out
            else:
                hf_dev = self.act_buffer()
                ff.featfix_debug_block(self.ctx, i, l, u, hf_dev, self.cond)
                torch.cuda.synchronize()
            steps = [r for r in wl.refresh if r <= i]
            if site_updates_history:
                steps += [s for (s, ll) in wl.sites if ll == l and s < i]
            steps = sorted(steps, reverse=True)[:len(hist)]
            u64, hf = self.to_logical(u), self.to_logical(hf_dev)
            h = [(s, self.to_logical(r)) for s, r in zip(steps, hist)]
            # Eq. 4 compares block outputs; in bf16 mode they are stored in
            # bf16, so the draft enters the discrepancy as it would be
            # forwarded: rounded to the model dtype
            hd = oracle.draft.draft(u64, h, i, wl.K)
            if sh.dtype == "bf16":
                hd = torch.from_numpy(hd).to(torch.bfloat16).double().numpy()
            for key, fn in (("rel_l1", oracle.featfix.rel_l1), ("rel_l2", oracle.featfix.rel_l2)):
                ref = fn(hd, hf)
                err = abs(got[(i, l)][key] - ref) / ref
                worst = max(worst, err)
                assert err <= tol, ((i, l), key, got[(i, l)][key], ref)
        return worst

    def close(self):
        ff.featfix_destroy(self.ctx)
        self.ctx = None

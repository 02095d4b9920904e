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


def log_close(got, ref, dtype):
    """Logged discrepancy (Eq. 4 / rel-L2) of a free-running trajectory.

    fp32: relative 1e-3.  bf16: h_d and h_f are stored in bf16, whose unit
    roundoff 2^-8 adds rounding noise of that relative size to ||h_d - h_f||
    -- as large as the discrepancy itself at these sites -- so the bound is
    5% of the value plus 2^-8 absolute."""
    if dtype == "f32":
        return abs(got - ref) <= 1e-3 * abs(ref)
    return abs(got - ref) <= 0.05 * abs(ref) + 2.0 ** -8


class Case:
    """One model + schedule on cuda:0 with the matching oracle inputs."""

    def __init__(self, wl, seed=0, weights_on_gpu=False):
        self.wl = wl
        self.sh = sh = wl.shape
        self.dev = torch.device("cuda:0")
        if weights_on_gpu:
            self.w = syn.make_weights(sh, seed=seed, device=self.dev)
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

    def close(self):
        ff.featfix_destroy(self.ctx)
        self.ctx = None

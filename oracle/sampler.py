"""Samplers and classifier-free guidance, float64.

The paper runs its method inside diffusion, flow-matching and rectified-flow
samplers (Section 3.1) without changing them; the concrete updates used here:

* Euler flow matching / rectified flow: sigma_i = 1 - i / N for i = 0..N,
  model time t_i = 1000 * sigma_i, update x <- x + (sigma_{i+1} - sigma_i) * v.
* DDIM (eta = 0) over a 1000-step linear beta schedule (1e-4 .. 0.02):
  the N steps visit tau_i = 1000 - (1000 / N) * (i + 1), i.e. 980 .. 0 for
  N = 50; alpha_bar after the last step is 1.  With eps from the model,
  x0 = (x - sqrt(1 - a_t) eps) / sqrt(a_t) and
  x <- sqrt(a_prev) x0 + sqrt(1 - a_prev) eps.  A learned-sigma head carries
  2 * C_in channels, of which the first C_in are eps.
* Guidance: the model batch is [conditional half ; unconditional half] and
  the guided output is out_u + s * (out_c - out_u).

Test infrastructure only.
"""

import numpy as np

DDIM_T = 1000


def euler_sigmas(steps):
    return np.array([1.0 - i / steps for i in range(steps + 1)], dtype=np.float64)


def ddim_alpha_bar():
    betas = np.linspace(1e-4, 0.02, DDIM_T, dtype=np.float64)
    return np.cumprod(1.0 - betas)


def ddim_timesteps(steps):
    stride = DDIM_T // steps
    return [DDIM_T - stride * (i + 1) for i in range(steps)]


def model_time(sampler, steps, i):
    """Timestep value fed to the model's sinusoidal embedding at step i."""
    if sampler == "euler":
        return 1000.0 * euler_sigmas(steps)[i]
    return float(ddim_timesteps(steps)[i])


def guide(out, batch, cfg, scale):
    """Classifier-free guidance over the model batch [cond ; uncond]."""
    if not cfg:
        return out
    oc, ou = out[:batch], out[batch:]
    return ou + scale * (oc - ou)


def euler_update(x, v, steps, i):
    sig = euler_sigmas(steps)
    return x + (sig[i + 1] - sig[i]) * v


def ddim_update(x, eps, steps, i):
    ab = ddim_alpha_bar()
    ts = ddim_timesteps(steps)
    a_t = ab[ts[i]]
    a_prev = ab[ts[i + 1]] if i + 1 < steps else 1.0
    x0 = (x - np.sqrt(1.0 - a_t) * eps) / np.sqrt(a_t)
    return np.sqrt(a_prev) * x0 + np.sqrt(1.0 - a_prev) * eps


def step_update(shape, x, model_out, steps, i):
    """Guidance then the sampler update of the latent x [B_lat, ...]."""
    g = guide(model_out, shape.batch, shape.cfg, shape.cfg_scale)
    if shape.sampler == "ddim":
        return ddim_update(x, g[:, :shape.in_ch], steps, i)
    return euler_update(x, g[:, :shape.in_ch], steps, i)

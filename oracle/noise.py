"""Seeded initial latent: SplitMix64 counters -> uniforms -> Box-Muller normals.

SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom number
generators", OOPSLA 2014) as a counter-based generator: the k-th 64-bit word
of stream ``seed`` is mix(seed + (k + 1) * 0x9E3779B97F4A7C15) with the
published finaliser
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9
    z = (z ^ (z >> 27)) * 0x94D049BB133111EB
    z =  z ^ (z >> 31)
(all mod 2^64).  A word maps to the open unit interval as
((w >> 11) + 0.5) * 2^-53.  Normal pair m uses words 2m and 2m + 1:
r = sqrt(-2 ln u_{2m}), phi = 2 pi u_{2m+1},
n_{2m} = r cos phi, n_{2m+1} = r sin phi (Box and Muller, 1958), computed in
float64 and rounded to float32.  Element n of the flattened latent takes n_n.

Test infrastructure only.
"""

import numpy as np

GOLDEN = np.uint64(0x9E3779B97F4A7C15)
M1 = np.uint64(0xBF58476D1CE4E5B9)
M2 = np.uint64(0x94D049BB133111EB)


def splitmix64_words(seed, count):
    """Words 0 .. count-1 of the counter-based SplitMix64 stream ``seed``."""
    k = np.arange(1, count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(seed) + k * GOLDEN
        z = (z ^ (z >> np.uint64(30))) * M1
        z = (z ^ (z >> np.uint64(27))) * M2
        z = z ^ (z >> np.uint64(31))
    return z


def normals(seed, count):
    """``count`` N(0, 1) samples as float32."""
    pairs = (count + 1) // 2
    w = splitmix64_words(seed, 2 * pairs)
    u = ((w >> np.uint64(11)).astype(np.float64) + 0.5) * (2.0 ** -53)
    u1, u2 = u[0::2], u[1::2]
    r = np.sqrt(-2.0 * np.log(u1))
    phi = 2.0 * np.pi * u2
    out = np.empty(2 * pairs, dtype=np.float64)
    out[0::2] = r * np.cos(phi)
    out[1::2] = r * np.sin(phi)
    return out[:count].astype(np.float32)


def initial_latent(seed, shape):
    """x_T for ``shape`` ([B, C_in, H, W] or [B, C_in, F, H, W]) from ``seed``."""
    dims = (shape.batch, shape.in_ch) + ((shape.lat_f,) if shape.lat_f > 0 else ()) + (shape.lat_h, shape.lat_w)
    return normals(seed, int(np.prod(dims))).reshape(dims)

"""FLOP accounting of the exact blocks (Table 1 reports FLOPs per method).

One multiply-add counts 2 FLOPs.  Per exact block: the four linear layers of
each stream (modulation GEMVs excluded) plus non-causal attention,
4 * N^2 * d * H per sample (q k^T and p v).

Test infrastructure only.
"""


def block_flops(shape, layer):
    C, M = shape.hidden, shape.mlp
    B = shape.batch * (2 if shape.cfg else 1)
    H, d = shape.heads, shape.head_dim
    if shape.arch == "dit":
        N = shape.img_tokens
        lin = 2 * B * N * (C * 3 * C + C * C + C * M + M * C)
        return lin + 4 * B * N * N * d * H
    N = shape.img_tokens + shape.txt_tokens
    if layer < shape.n_dual:
        lin = 2 * B * N * (C * 3 * C + C * C + C * M + M * C)
    else:
        lin = 2 * B * N * (C * (3 * C + M) + (C + M) * C)
    return lin + 4 * B * N * N * d * H


def step_flops(shape):
    """All blocks of one denoising step."""
    L = shape.n_dual + shape.n_single if shape.arch == "mmdit" else shape.n_dual
    return sum(block_flops(shape, l) for l in range(L))

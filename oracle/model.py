"""Exact transformer blocks of the denoiser, float64 (FeatFix Eq. 1).

The paper writes the exact block output as h^f = B_l(u; t, c) (Eq. 1) and
names an adaLN-modulated attention + MLP block; the layer-level details it
leaves open are fixed here as follows (the readings are listed in the design
notes):

* LayerNorm without affine parameters, eps = 1e-6.
* modulate(x, shift, scale) = x * (1 + scale) + shift, per sample.
* GELU with the tanh approximation.
* Non-causal softmax(q k^T / sqrt(d)) v attention.
* Modulation vectors are Linear(SiLU(c)); chunk order
  (shift1, scale1, gate1, shift2, scale2, gate2) for a two-branch block,
  (shift, scale, gate) for a single-stream block, (shift, scale) for the
  final layer.
* qkv columns are [q | k | v], head h owning columns h*d .. h*d+d-1 of each.
* MMDiT: text tokens come first, image tokens after; rotary embedding is
  applied to image-token queries and keys only, interleaved pairs
  (2j, 2j+1), theta = 10000, per-axis frequency theta^(-2j / d_axis).

Shapes: token tensors are [B, N, C] (logical layout, text before image).
Weights are a dict name -> float64 array, nn.Linear convention
(weight [out, in], y = x W^T + b).

Test infrastructure only: never imported by the product path.
"""

import numpy as np

LN_EPS = 1e-6
T_FREQ_DIM = 256
ROPE_THETA = 10000.0


# ----------------------------------------------------------------------------
# primitives
# ----------------------------------------------------------------------------

def layer_norm(x):
    """LayerNorm over the last axis, no affine, eps = 1e-6."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + LN_EPS)


def modulate(x, shift, scale):
    """adaLN modulation x * (1 + scale) + shift; shift/scale are [B, C]."""
    return x * (1.0 + scale[:, None, :]) + shift[:, None, :]


def gelu_tanh(x):
    """GELU, tanh approximation."""
    return 0.5 * x * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3)))


def silu(x):
    return x / (1.0 + np.exp(-x))


def linear(x, w, b):
    """nn.Linear: y = x W^T + b with W [out, in]."""
    return x @ w.T + b


def attention(q, k, v):
    """Non-causal softmax(q k^T / sqrt(d)) v over [B, H, N, d] tensors.

    Loops over (batch, head) so one score matrix is alive at a time.
    """
    B, H, N, d = q.shape
    out = np.empty_like(q)
    scale = 1.0 / np.sqrt(d)
    for b in range(B):
        for h in range(H):
            s = (q[b, h] @ k[b, h].T) * scale
            s = s - s.max(axis=-1, keepdims=True)
            p = np.exp(s)
            p /= p.sum(axis=-1, keepdims=True)
            out[b, h] = p @ v[b, h]
    return out


def split_heads(x, heads):
    """[B, N, H*d] -> [B, H, N, d]."""
    B, N, C = x.shape
    return x.reshape(B, N, heads, C // heads).transpose(0, 2, 1, 3)


def merge_heads(x):
    """[B, H, N, d] -> [B, N, H*d]."""
    B, H, N, d = x.shape
    return x.transpose(0, 2, 1, 3).reshape(B, N, H * d)


# ----------------------------------------------------------------------------
# rotary position embedding (MMDiT image tokens)
# ----------------------------------------------------------------------------

def rope_axes(head_dim, rope_dims):
    """Per-axis rotary widths: 2-D splits d into halves, 3-D into 1/8, 7/16, 7/16."""
    if rope_dims == 2:
        return (head_dim // 2, head_dim // 2)
    if rope_dims == 3:
        t = head_dim // 8
        hw = (head_dim - t) // 2
        return (t, hw, head_dim - t - hw)
    raise ValueError("rope_dims must be 2 or 3")


def rope_angles(positions, axes):
    """Angles [N, d/2] for integer positions [N, n_axes] and axis widths.

    Pair j of axis a (width d_a) turns by pos_a * theta^(-2j/d_a).
    """
    cols = []
    for a, da in enumerate(axes):
        j = np.arange(da // 2, dtype=np.float64)
        freq = ROPE_THETA ** (-2.0 * j / da)
        cols.append(positions[:, a:a + 1].astype(np.float64) * freq[None, :])
    return np.concatenate(cols, axis=1)


def apply_rope(x, ang):
    """Rotate interleaved pairs (2j, 2j+1) of x [B, H, N, d] by ang [N, d/2]."""
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., 0::2], x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = x1 * c - x2 * s
    out[..., 1::2] = x1 * s + x2 * c
    return out


def image_positions(grid):
    """Integer positions of image tokens in row-major order of the patch grid."""
    idx = np.indices(grid).reshape(len(grid), -1).T
    return idx


# ----------------------------------------------------------------------------
# conditioning and token embedding
# ----------------------------------------------------------------------------

def timestep_sinusoid(t, dim=T_FREQ_DIM, max_period=10000.0):
    """Sinusoidal timestep features, [cos | sin] halves, frequencies
    max_period^(-k/half) for k = 0..half-1."""
    half = dim // 2
    freqs = np.exp(-np.log(max_period) * np.arange(half, dtype=np.float64) / half)
    args = float(t) * freqs
    return np.concatenate([np.cos(args), np.sin(args)])


def cond_vector(W, t, labels=None, batch=1):
    """c = MLP(sinusoid(t)) (+ label embedding for class-conditional models).

    Returns [B, C].
    """
    s = timestep_sinusoid(t)
    e = linear(silu(linear(s, W["t_fc1.w"], W["t_fc1.b"])), W["t_fc2.w"], W["t_fc2.b"])
    c = np.repeat(e[None, :], batch, axis=0)
    if labels is not None:
        c = c + W["y_emb"][np.asarray(labels)]
    return c


def sincos_pos_2d(C, gh, gw):
    """Fixed 2-D sin-cos position embedding [gh*gw, C].

    The first C/2 channels encode the patch row, the last C/2 the patch
    column; each half is [sin(pos * w_k) | cos(pos * w_k)] with
    w_k = 10000^(-k / (C/4)), k = 0 .. C/4 - 1.
    """
    q = C // 4
    w = 10000.0 ** (-np.arange(q, dtype=np.float64) / q)
    rows, cols = np.meshgrid(np.arange(gh), np.arange(gw), indexing="ij")
    rows = rows.reshape(-1).astype(np.float64)
    cols = cols.reshape(-1).astype(np.float64)
    er = np.concatenate([np.sin(rows[:, None] * w), np.cos(rows[:, None] * w)], axis=1)
    ec = np.concatenate([np.sin(cols[:, None] * w), np.cos(cols[:, None] * w)], axis=1)
    return np.concatenate([er, ec], axis=1)


def patch_grid(shape):
    """Patch grid (tuple) and patch volume for a model shape."""
    if shape.lat_f > 0:
        return (shape.lat_f // shape.patch_t, shape.lat_h // shape.patch, shape.lat_w // shape.patch), \
            shape.patch_t * shape.patch * shape.patch
    return (shape.lat_h // shape.patch, shape.lat_w // shape.patch), shape.patch * shape.patch


def patchify(x, shape):
    """Latent -> [B, N_img, C_in * P]; tokens row-major over the patch grid,
    features ordered (channel, patch offsets)."""
    p = shape.patch
    if shape.lat_f > 0:
        B, Ci, F, H, Wd = x.shape
        pt = shape.patch_t
        y = x.reshape(B, Ci, F // pt, pt, H // p, p, Wd // p, p)
        y = y.transpose(0, 2, 4, 6, 1, 3, 5, 7)
        return y.reshape(B, (F // pt) * (H // p) * (Wd // p), Ci * pt * p * p)
    B, Ci, H, Wd = x.shape
    y = x.reshape(B, Ci, H // p, p, Wd // p, p).transpose(0, 2, 4, 1, 3, 5)
    return y.reshape(B, (H // p) * (Wd // p), Ci * p * p)


def unpatchify(y, shape, ch):
    """Inverse of ``patchify`` with ``ch`` output channels."""
    p = shape.patch
    B = y.shape[0]
    if shape.lat_f > 0:
        pt = shape.patch_t
        F, H, Wd = shape.lat_f, shape.lat_h, shape.lat_w
        z = y.reshape(B, F // pt, H // p, Wd // p, ch, pt, p, p)
        z = z.transpose(0, 4, 1, 5, 2, 6, 3, 7)
        return z.reshape(B, ch, F, H, Wd)
    H, Wd = shape.lat_h, shape.lat_w
    z = y.reshape(B, H // p, Wd // p, ch, p, p).transpose(0, 3, 1, 4, 2, 5)
    return z.reshape(B, ch, H, Wd)


def embed_tokens(W, shape, x_model, txt=None):
    """Block-0 input: DiT = patch embed + 2-D sin-cos position; MMDiT =
    [text tokens ; patch embed]."""
    if shape.arch == "dit":
        grid, _ = patch_grid(shape)
        tok = linear(patchify(x_model, shape), W["x_emb.w"], W["x_emb.b"])
        return tok + sincos_pos_2d(shape.hidden, grid[0], grid[1])[None]
    img = linear(patchify(x_model, shape), W["img_in.w"], W["img_in.b"])
    return np.concatenate([np.asarray(txt, dtype=np.float64), img], axis=1)


def final_layer(W, shape, tok, c):
    """LN + modulate with (shift, scale) = Linear(SiLU(c)), Linear to patch
    features, unpatchify.  MMDiT keeps the image tokens only."""
    if shape.arch == "mmdit":
        tok = tok[:, shape.txt_tokens:]
    m = linear(silu(c), W["final.mod.w"], W["final.mod.b"])
    shift, scale = np.split(m, 2, axis=-1)
    y = linear(modulate(layer_norm(tok), shift, scale), W["final.lin.w"], W["final.lin.b"])
    return unpatchify(y, shape, shape.out_ch)


# ----------------------------------------------------------------------------
# exact blocks B_l (Eq. 1)
# ----------------------------------------------------------------------------

def dit_block(W, pre, u, c, heads):
    """DiT adaLN block: attention branch then MLP branch, each gated."""
    m = linear(silu(c), W[pre + "mod.w"], W[pre + "mod.b"])
    sh1, sc1, g1, sh2, sc2, g2 = np.split(m, 6, axis=-1)
    a = modulate(layer_norm(u), sh1, sc1)
    qkv = linear(a, W[pre + "qkv.w"], W[pre + "qkv.b"])
    q, k, v = np.split(qkv, 3, axis=-1)
    o = merge_heads(attention(split_heads(q, heads), split_heads(k, heads), split_heads(v, heads)))
    u1 = u + g1[:, None, :] * linear(o, W[pre + "proj.w"], W[pre + "proj.b"])
    a2 = modulate(layer_norm(u1), sh2, sc2)
    y = linear(gelu_tanh(linear(a2, W[pre + "fc1.w"], W[pre + "fc1.b"])), W[pre + "fc2.w"], W[pre + "fc2.b"])
    return u1 + g2[:, None, :] * y


def _rope_qk(q, k, n_txt, ang):
    """Apply the rotary embedding to the image part (tokens >= n_txt)."""
    if ang is None:
        return q, k
    q = q.copy()
    k = k.copy()
    q[:, :, n_txt:] = apply_rope(q[:, :, n_txt:], ang)
    k[:, :, n_txt:] = apply_rope(k[:, :, n_txt:], ang)
    return q, k


def mmdit_dual_block(W, pre, u, c, heads, n_txt, ang):
    """Two-stream block: per-stream modulation, qkv, projection and MLP;
    joint attention over [text ; image]."""
    txt, img = u[:, :n_txt], u[:, n_txt:]
    mi = np.split(linear(silu(c), W[pre + "img_mod.w"], W[pre + "img_mod.b"]), 6, axis=-1)
    mt = np.split(linear(silu(c), W[pre + "txt_mod.w"], W[pre + "txt_mod.b"]), 6, axis=-1)
    qkv_i = linear(modulate(layer_norm(img), mi[0], mi[1]), W[pre + "img_qkv.w"], W[pre + "img_qkv.b"])
    qkv_t = linear(modulate(layer_norm(txt), mt[0], mt[1]), W[pre + "txt_qkv.w"], W[pre + "txt_qkv.b"])
    qkv = np.concatenate([qkv_t, qkv_i], axis=1)
    q, k, v = (split_heads(z, heads) for z in np.split(qkv, 3, axis=-1))
    q, k = _rope_qk(q, k, n_txt, ang)
    o = merge_heads(attention(q, k, v))
    o_t, o_i = o[:, :n_txt], o[:, n_txt:]
    img = img + mi[2][:, None] * linear(o_i, W[pre + "img_proj.w"], W[pre + "img_proj.b"])
    txt = txt + mt[2][:, None] * linear(o_t, W[pre + "txt_proj.w"], W[pre + "txt_proj.b"])
    yi = linear(gelu_tanh(linear(modulate(layer_norm(img), mi[3], mi[4]), W[pre + "img_fc1.w"], W[pre + "img_fc1.b"])),
                W[pre + "img_fc2.w"], W[pre + "img_fc2.b"])
    yt = linear(gelu_tanh(linear(modulate(layer_norm(txt), mt[3], mt[4]), W[pre + "txt_fc1.w"], W[pre + "txt_fc1.b"])),
                W[pre + "txt_fc2.w"], W[pre + "txt_fc2.b"])
    img = img + mi[5][:, None] * yi
    txt = txt + mt[5][:, None] * yt
    return np.concatenate([txt, img], axis=1)


def mmdit_single_block(W, pre, u, c, heads, n_txt, ang):
    """Single-stream block: one modulation, linear1 -> [qkv | mlp], joint
    attention, linear2 over [attention | GELU(mlp)], one gate."""
    C = u.shape[-1]
    sh, sc, g = np.split(linear(silu(c), W[pre + "mod.w"], W[pre + "mod.b"]), 3, axis=-1)
    y = linear(modulate(layer_norm(u), sh, sc), W[pre + "lin1.w"], W[pre + "lin1.b"])
    qkv, mlp = y[..., :3 * C], y[..., 3 * C:]
    q, k, v = (split_heads(z, heads) for z in np.split(qkv, 3, axis=-1))
    q, k = _rope_qk(q, k, n_txt, ang)
    o = merge_heads(attention(q, k, v))
    out = linear(np.concatenate([o, gelu_tanh(mlp)], axis=-1), W[pre + "lin2.w"], W[pre + "lin2.b"])
    return u + g[:, None, :] * out


def block_prefix(shape, layer):
    if shape.arch == "dit":
        return "blk%d." % layer
    if layer < shape.n_dual:
        return "dual%d." % layer
    return "single%d." % (layer - shape.n_dual)


def rope_table(shape):
    """Angles for the image tokens of an MMDiT model (None for DiT)."""
    if shape.arch != "mmdit" or shape.rope_dims == 0:
        return None
    grid, _ = patch_grid(shape)
    return rope_angles(image_positions(grid), rope_axes(shape.head_dim, shape.rope_dims))


def exact_block(W, shape, layer, u, c, ang=None):
    """h^f = B_l(u; t, c) (Eq. 1) for layer ``layer`` of ``shape``."""
    pre = block_prefix(shape, layer)
    if shape.arch == "dit":
        return dit_block(W, pre, u, c, shape.heads)
    if ang is None:
        ang = rope_table(shape)
    if layer < shape.n_dual:
        return mmdit_dual_block(W, pre, u, c, shape.heads, shape.txt_tokens, ang)
    return mmdit_single_block(W, pre, u, c, shape.heads, shape.txt_tokens, ang)

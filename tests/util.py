"""Small hand-built assets for tests (no randomness unless a seed is given)."""
import numpy as np

from paper_2608_27888_gb300 import workloads as W

QD = W.QUERY_DTYPE


def half_bits(values):
    return np.asarray(values, dtype=np.float16).view(np.uint16)


def tiny_assets(level_dims, num_mips=1, channels=8, latents=None, hidden=16, out_dim=4,
                layers=2, num_decoders=1, set_to_decoder=None, weights=None, address_mode=0,
                num_sets=1, pe_frequencies=0, activation=0, leaky_slope=0.01):
    """Assets with explicit latents (float array, rounded to fp16) and weights."""
    dims, offs, total = W.pyramid_layout(num_sets, level_dims, num_mips)
    L = dims.shape[1]
    if latents is None:
        latents = np.zeros(total * channels, dtype=np.float32)
    lat = half_bits(np.asarray(latents, dtype=np.float32).reshape(-1))
    assert lat.size == total * channels
    in_dim = L * channels + 4 * pe_frequencies
    per = hidden * in_dim + hidden + (layers - 1) * (hidden * hidden + hidden) + out_dim * hidden + out_dim
    if weights is None:
        weights = np.zeros((num_decoders, per), dtype=np.float32)
    if set_to_decoder is None:
        set_to_decoder = np.zeros(num_sets, dtype=np.uint32)
    return W.Assets(num_sets=num_sets, num_levels=L, num_mips=num_mips, channels=channels,
                    level_dims=dims, latent_offsets=offs, latents=lat, num_decoders=num_decoders,
                    in_dim=in_dim, hidden=hidden, num_hidden_layers=layers, out_dim=out_dim,
                    weights=np.asarray(weights, dtype=np.float32).reshape(num_decoders, per),
                    set_to_decoder=np.asarray(set_to_decoder, dtype=np.uint32),
                    address_mode=address_mode, pe_frequencies=pe_frequencies,
                    activation=activation, leaky_slope=leaky_slope)


def queries(rows):
    q = np.zeros(len(rows), dtype=QD)
    for i, (s, u, v, lod) in enumerate(rows):
        q[i] = (s, u, v, lod)
    return q


def split_weights(a, d=0):
    """Views W1, b1, [W_l, b_l]..., Wout, bout of decoder d (row-major [out][in])."""
    p = a.weights[d]
    H, I, C = a.hidden, a.in_dim, a.out_dim
    out, o = [], 0

    def take(r, c):
        nonlocal o
        m = p[o:o + r * c].reshape(r, c) if c else p[o:o + r]
        o += r * c if c else r
        return m
    out.append(take(H, I)); out.append(take(H, 0))
    for _ in range(a.num_hidden_layers - 1):
        out.append(take(H, H)); out.append(take(H, 0))
    out.append(take(C, H)); out.append(take(C, 0))
    assert o == p.size
    return out

"""Seeded synthetic workloads for the latent cache and attention.

This module draws inputs only; it holds none of the method's arithmetic, so
both the CUDA path and the float64 CPU checker can consume what it returns.
All values are drawn in float64 from ``numpy.random.default_rng(seed)`` and
rounded once to bfloat16; both sides see the same bfloat16 bits.

Shapes follow the Wan2.1-1.3B backbone the paper builds on (Sec. 4.1,
App. D.1-D.2): hidden 1536, 12 heads of 128, d_c = 192, d_r = 32,
d_q = 768, latent frames of 30 x 52 = 1560 tokens, chunks of 3 latent frames,
a window of 21 latent frames. Distributions: activations x ~ N(0, 1); every
projection W ~ N(0, 1/fan_in); cached latents c ~ N(0, 1) (what an RMSNorm'd
latent looks like); positional keys and queries ~ N(0, 1); absorbed content
queries q_c ~ N(0, d_nope / d_c), the variance of (W_up^K)^T W_up^Q c^Q under
that weight init with a unit-RMS query latent.
"""

from dataclasses import dataclass, replace

import numpy as np
import torch

__all__ = ["Workload", "WORKLOADS", "workload", "bf16", "draw_layer_weights",
           "draw_tokens", "grid_positions", "frame_coords", "draw_queries", "draw_cache_rows",
           "unit_vectors", "fill_normal_"]


@dataclass(frozen=True)
class Workload:
    name: str
    hidden: int = 1536
    heads: int = 12
    head_dim: int = 128
    d_c: int = 192
    d_r: int = 32
    d_q: int = 768
    rope_pairs: tuple = (6, 5, 5)          # complex pairs over (t, h, w)
    rope_axis_dims: tuple = (44, 42, 42)   # band widths of the 128-channel split
    rope_theta: float = 10000.0
    rope_table_len: int = 1024
    grid_h: int = 30
    grid_w: int = 52
    window_frames: int = 21
    chunk_frames: int = 3
    batch: int = 1
    last_frame: int = 21                  # frames_written after the timed chunk
    rms_eps: float = 1e-6
    layers: int = 1                       # attention layers per benchmark step
    sink_frames: int = 0                  # frames never evicted (long-rollout window)

    @property
    def tokens_per_frame(self):
        return self.grid_h * self.grid_w

    @property
    def slots(self):
        return self.tokens_per_frame * self.window_frames

    @property
    def chunk_tokens(self):
        return self.tokens_per_frame * self.chunk_frames

    def with_(self, **kw):
        return replace(self, **kw)


WORKLOADS = {
    # 8x8 latent grid, one-frame chunk, 3 cached frames + itself; RoPE
    # channels 8/12/12 over (t, h, w)
    "tiny": Workload("tiny", rope_pairs=(4, 6, 6), grid_h=8, grid_w=8,
                     window_frames=4, chunk_frames=1, last_frame=4),
    # Wan2.1-1.3B layer: 4680-token chunk against a full 21-frame window,
    # the paper's (6, 5, 5) RoPE pairs
    "wan": Workload("wan"),
    # a full denoising step of the 30-block backbone: one Wan layer per block
    "wan30": Workload("wan30", layers=30),
    # batch 4, positions advancing to latent frame 960 in a 21-frame ring
    "rollout": Workload("rollout", batch=4, last_frame=960),
    # the paper's long-rollout window: 1 sink frame + the 6 newest frames,
    # k^R cached unrotated and re-indexed per window, frames to 960, batch 4
    "sink": Workload("sink", batch=4, window_frames=7, sink_frames=1, last_frame=960),
}


def workload(name, **overrides):
    w = WORKLOADS[name]
    return w.with_(**overrides) if overrides else w


def bf16(a):
    """float64 array -> bfloat16 CPU tensor (round to nearest even)."""
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)


def _normal(rng, shape, std):
    return rng.standard_normal(shape) * std


def draw_layer_weights(w, seed):
    """All projections of one VideoMLA layer, bfloat16, W ~ N(0, 1/fan_in).

    Shapes (App. D.2): w_dkv [d_c, d], w_kr [d_r, d], w_dq [d_q, d],
    w_uk [H, d_nope, d_c], w_uv [H, d_h, d_c], w_uq [H, d_nope, d_q],
    w_qr [H, d_r, d_q], w_o [d, H d_h]; gamma_kv [d_c], gamma_q [d_q] = 1.
    """
    rng = np.random.default_rng(seed)
    d, H, dh, dc, dr, dq = w.hidden, w.heads, w.head_dim, w.d_c, w.d_r, w.d_q
    dn = dh - dr
    out = {
        "w_dkv": _normal(rng, (dc, d), d ** -0.5),
        "w_kr": _normal(rng, (dr, d), d ** -0.5),
        "w_dq": _normal(rng, (dq, d), d ** -0.5),
        "w_uk": _normal(rng, (H, dn, dc), dc ** -0.5),
        "w_uv": _normal(rng, (H, dh, dc), dc ** -0.5),
        "w_uq": _normal(rng, (H, dn, dq), dq ** -0.5),
        "w_qr": _normal(rng, (H, dr, dq), dq ** -0.5),
        "w_o": _normal(rng, (d, H * dh), (H * dh) ** -0.5),
        "gamma_kv": np.ones(dc),
        "gamma_q": np.ones(dq),
    }
    return {k: bf16(v) for k, v in out.items()}


def draw_tokens(w, n_tokens, seed, batch=None):
    """Activations x [B, n_tokens, hidden] ~ N(0, 1), bfloat16."""
    rng = np.random.default_rng(seed)
    B = w.batch if batch is None else batch
    return bf16(rng.standard_normal((B, n_tokens, w.hidden)))


def grid_positions(w, first_frame, n_frames, batch=None):
    """(t, h, w) of every token of frames first_frame .. first_frame+n_frames-1.

    Tokens of a latent frame are in raster order over the grid_h x grid_w grid;
    t is the absolute latent-frame index. int32 [B, n_frames * T, 3].
    """
    B = w.batch if batch is None else batch
    t = np.repeat(np.arange(first_frame, first_frame + n_frames), w.tokens_per_frame)
    hh = np.tile(np.repeat(np.arange(w.grid_h), w.grid_w), n_frames)
    ww = np.tile(np.arange(w.grid_w), w.grid_h * n_frames)
    pos = np.stack([t, hh, ww], axis=-1).astype(np.int32)
    return torch.from_numpy(np.repeat(pos[None], B, axis=0))


def frame_coords(w):
    """(h, w) of token k of a latent frame, raster order: int32 [T, 2]."""
    hh = np.repeat(np.arange(w.grid_h), w.grid_w)
    ww = np.tile(np.arange(w.grid_w), w.grid_h)
    return torch.from_numpy(np.stack([hh, ww], axis=-1).astype(np.int32))


def draw_queries(w, n_tokens, seed, batch=None, qc_std=None, qr_std=1.0, as_float64=False):
    """Absorbed content queries q_c [B, n, H, d_c] and unrotated q_r [B, n, H, d_r].

    q_c ~ N(0, qc_std^2) with qc_std = sqrt(d_nope / d_c) by default; q_r ~
    N(0, qr_std^2). as_float64 returns the float64 draws before rounding (for
    callers that build structured inputs and round them once themselves)."""
    rng = np.random.default_rng(seed)
    B = w.batch if batch is None else batch
    dn = w.head_dim - w.d_r
    q_c = _normal(rng, (B, n_tokens, w.heads, w.d_c),
                  (dn / w.d_c) ** 0.5 if qc_std is None else qc_std)
    q_r = _normal(rng, (B, n_tokens, w.heads, w.d_r), qr_std)
    if as_float64:
        return q_c, q_r
    return bf16(q_c), bf16(q_r)


def unit_vectors(n, d, seed):
    """n random directions in R^d (rows of unit length), float64."""
    rng = np.random.default_rng(seed)
    u = rng.standard_normal((n, d))
    return u / np.linalg.norm(u, axis=1, keepdims=True)


def draw_cache_rows(w, n_rows, seed, batch=None, as_float64=False):
    """Cache contents c [B, n, d_c] ~ N(0,1) and rotated keys k [B, n, d_r] ~ N(0,1)."""
    rng = np.random.default_rng(seed)
    B = w.batch if batch is None else batch
    c, k = rng.standard_normal((B, n_rows, w.d_c)), rng.standard_normal((B, n_rows, w.d_r))
    if as_float64:
        return c, k
    return bf16(c), bf16(k)


def fill_normal_(t, seed, std=1.0):
    """Fill a (CUDA) tensor in place with N(0, std^2) draws of a seeded torch
    generator on its device, rounded once to the tensor's dtype: inputs of
    batches too large to draw on the host (both sides read the same values
    back)."""
    g = torch.Generator(device=t.device).manual_seed(seed)
    t.normal_(0.0, std, generator=g)
    return t

"""Float64 CPU oracle for VideoMLA's latent KV cache and attention.

TEST INFRASTRUCTURE ONLY. Nothing in the product path imports this module:
only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may call it. It shares no code with the CUDA path (no table
builders, no constants, no helpers). Every function takes plain float64
NumPy arrays and is written to be checked against the paper by eye:
no blocking, no fusion, no reordering beyond what the cited passage states.

Paper: "VideoMLA" (arXiv 2605.30351).

  * Sec. 3.1, Eq. (ckv)          c^KV = W_dn^KV x
  * App. D.2 (VideoMLA block)    RMSNorm on c^KV and on c^Q before up-projection
  * Sec. 3.1, Eq. (reconstruct)  k^nope_h = W_up,h^K c^KV ,  v_h = W_up,h^V c^KV
  * Sec. 3.1, Eqs. (cq), (qnope) c^Q = W_dn^Q x ,  q^nope_h = W_up,h^Q c^Q
  * Sec. 3.2, Eqs. (krope), (qrope)  k^R = W_R^K x ; q^R_h = W_R,h^Q c^Q ; RoPE_3D
  * Sec. 3.3, Eq. (score)        (q^nope.k^nope + q^rope.k^rope) / sqrt(d_nope + d_rope)
  * App. D.4                     chunk-causal mask, sliding window, FIFO eviction
  * App. E, Eqs. (absorb-q), (absorb-v)  absorbed (latent) inference form

Readings taken where the paper is silent (each one is listed in the design
notes of the repository):

  R1  3D-RoPE frequencies. Pair i of axis a (a in t, h, w) uses the inverse
      frequency theta^(-2 i / D_a), i = 0 .. n_a - 1 (the highest-frequency
      bands of that axis), where D_a is the channel width of that axis in the
      backbone's 128-channel head split (44 / 42 / 42) and theta = 10000.
      Complex pairs are adjacent channels (2p, 2p+1); the pair blocks are
      ordered t, h, w. PARITY UNPINNED for the frequency VALUES: the paper
      prints neither theta nor the axis widths, so only the structure (a
      rotation per pair, highest band first, exact relative-position
      property) is pinned by the tests.
  R2  The positional key is rotated when it is appended, with the absolute
      (t, h, w) position the caller gives. For a window of contiguous frames
      the scores depend only on position differences, so this equals
      rotating at use with window-relative coordinates (Sec. 3.2, App. D.5).
  R3  RMSNorm is applied at append and the cache stores the normalised
      latent; eps = 1e-6; gamma is an input (ones in synthetic runs).
  R4  The score scale is 1/sqrt(d_h) with d_h = d_nope + d_rope (Eq. score),
      for every d_c.
  R5  Ring slot of token k of latent frame f: (f mod W_frames) * T + k
      (FIFO eviction, App. D.4).
  R12 Long-rollout window (App. D.4): the first S latent frames (S = 1, the
      sink) stay for good, the other W - S slots-frames hold the newest
      W - S frames in FIFO order (W - S = 6), and the current chunk is among
      them (it is appended before attention). Token k of frame f sits at
      f * T + k for f < S, else (S + (f - S) mod (W - S)) * T + k; S = 0 is
      the plain ring of R5.
  R13 Window-relative RoPE (App. D.5): the cache keeps k^R unrotated; when a
      window is assembled its held frames are numbered 0, 1, ... in temporal
      order (sinks first) and that number is the temporal coordinate of their
      keys and of the queries of those frames; (h, w) stay as given. Before
      any eviction this is the absolute frame index.
"""

import math

import numpy as np

__all__ = [
    "RopeSpec",
    "rope_inv_freq",
    "rope3d",
    "rmsnorm",
    "ring_slot",
    "window_frames",
    "sink_ring_slot",
    "sink_window_frames",
    "window_local_time",
    "window_attention",
    "OracleCache",
    "cache_append",
    "softmax",
    "latent_attention",
    "reference_attention",
    "dense_attention",
    "absorb_query",
    "absorb_output",
    "absorbed_query_matrices",
    "absorbed_output_matrices",
    "per_head_output_from_latent",
    "cache_scalars_per_token",
    "dense_scalars_per_token",
    "latent_attention_flops",
]


# --------------------------------------------------------------------------
# 3D-RoPE  (Sec. 3.2; App. D.3; reading R1)
# --------------------------------------------------------------------------
class RopeSpec:
    """Which axis each complex pair rotates with, and at what frequency."""

    def __init__(self, pairs=(6, 5, 5), axis_dims=(44, 42, 42), theta=10000.0):
        self.pairs = tuple(int(p) for p in pairs)
        self.axis_dims = tuple(int(d) for d in axis_dims)
        self.theta = float(theta)

    @property
    def d_r(self):
        return 2 * sum(self.pairs)


def rope_inv_freq(spec):
    """Return (inv_freq[n_pairs], axis[n_pairs]) for the pairs in t, h, w order.

    Reading R1: the first n_a bands of axis a, theta^(-2 i / D_a).
    """
    inv = []
    axis = []
    for a in range(3):
        for i in range(spec.pairs[a]):
            inv.append(spec.theta ** (-2.0 * i / spec.axis_dims[a]))
            axis.append(a)
    return np.array(inv, dtype=np.float64), np.array(axis, dtype=np.int64)


def rope3d(v, pos, spec):
    """Rotate the complex pairs of v by the token's 3D position.

    v   : [..., d_r] float64, pairs are channels (2p, 2p+1)
    pos : [..., 3]   integer (t, h, w), broadcast against v's leading dims
    Pair p is multiplied by exp(i * pos[axis(p)] * inv_freq[p]) (Sec. 3.2).
    """
    v = np.asarray(v, dtype=np.float64)
    pos = np.asarray(pos)
    inv, axis = rope_inv_freq(spec)
    out = np.empty_like(v)
    for p in range(len(inv)):
        ang = pos[..., axis[p]].astype(np.float64) * inv[p]
        cs, sn = np.cos(ang), np.sin(ang)
        x0 = v[..., 2 * p]
        x1 = v[..., 2 * p + 1]
        out[..., 2 * p] = x0 * cs - x1 * sn
        out[..., 2 * p + 1] = x0 * sn + x1 * cs
    return out


# --------------------------------------------------------------------------
# RMSNorm (App. D.2; reading R3)
# --------------------------------------------------------------------------
def rmsnorm(v, gamma=None, eps=1e-6):
    """gamma * v / sqrt(mean(v^2) + eps) over the last axis."""
    v = np.asarray(v, dtype=np.float64)
    ms = np.mean(v * v, axis=-1, keepdims=True)
    out = v / np.sqrt(ms + eps)
    if gamma is not None:
        out = out * np.asarray(gamma, dtype=np.float64)
    return out


# --------------------------------------------------------------------------
# Sliding-window ring (App. D.4; reading R5)
# --------------------------------------------------------------------------
def ring_slot(frame, k, tokens_per_frame, window_frames):
    """Slot of token k of latent frame `frame` in the FIFO ring."""
    return (frame % window_frames) * tokens_per_frame + k


def window_frames(frames_written, window_frames):
    """Latent frames held once `frames_written` frames were appended in order."""
    first = max(0, frames_written - window_frames)
    return list(range(first, frames_written))


# --------------------------------------------------------------------------
# Sink + FIFO window and window-relative RoPE (App. D.4, D.5; R12, R13)
# --------------------------------------------------------------------------
def sink_ring_slot(frame, k, tokens_per_frame, window_frames, sink_frames):
    """Slot of token k of latent frame `frame` when the first `sink_frames`
    frames are kept for good and the later frames share the remaining
    window_frames - sink_frames frame slots in FIFO order (reading R12)."""
    if frame < sink_frames:
        return frame * tokens_per_frame + k
    local = window_frames - sink_frames
    return (sink_frames + (frame - sink_frames) % local) * tokens_per_frame + k


def sink_window_frames(frames_written, window_frames, sink_frames):
    """Frames held after `frames_written` in-order appends, in temporal order:
    the sink frames, then the newest window_frames - sink_frames frames."""
    sinks = list(range(min(sink_frames, frames_written)))
    first_local = max(sink_frames, frames_written - (window_frames - sink_frames))
    return sinks + list(range(first_local, frames_written))


def window_local_time(frame, frames_written, window_frames, sink_frames):
    """Temporal coordinate of a held frame inside the assembled window: its
    index among the held frames in temporal order (reading R13). Raises
    ValueError for a frame the window does not hold."""
    return sink_window_frames(frames_written, window_frames, sink_frames).index(frame)


class OracleCache:
    """Latent cache state: c [B, slots, d_c], k [B, slots, d_r] (rotated at
    append, or unrotated for the window path), the frame of every slot and
    the (t, h, w) each slot's token was appended with."""

    def __init__(self, batch, tokens_per_frame, window_frames, d_c, d_r, sink_frames=0):
        self.T = tokens_per_frame
        self.W = window_frames
        self.S = sink_frames
        slots = tokens_per_frame * window_frames
        self.c = np.zeros((batch, slots, d_c))
        self.kr = np.zeros((batch, slots, d_r))
        self.pos_of_slot = np.zeros((batch, slots, 3), dtype=np.int64)
        self.frame_of_slot = np.full(slots, -1, dtype=np.int64)
        self.frames_written = 0

    def held_frames(self):
        return sink_window_frames(self.frames_written, self.W, self.S)

    def valid_slots(self):
        """Slots that hold a frame of the current window (App. D.4)."""
        held = set(self.held_frames())
        return np.array([s for s in range(len(self.frame_of_slot))
                         if self.frame_of_slot[s] in held], dtype=np.int64)


def cache_append(cache, x, w_dkv, w_kr, pos, first_frame, n_frames,
                 gamma=None, eps=1e-6, use_rmsnorm=True, spec=None):
    """Write n_frames latent frames of tokens into the cache.

    x    : [B, n_frames*T, d] token activations
    w_dkv: [d_c, d]  joint KV down-projection      (Eq. ckv)
    w_kr : [d_r, d]  decoupled RoPE key projection (Eq. krope)
    pos  : [B, n_frames*T, 3] (t, h, w) of each token
    Stores c = RMSNorm(W_dkv x) (reading R3) and k = RoPE3D(W_kr x, pos)
    (reading R2), or k = W_kr x unrotated when spec is None (the paper's
    storage, App. D.5), at the FIFO slots of frames
    first_frame .. first_frame+n_frames-1 (readings R5, R12).
    """
    x = np.asarray(x, dtype=np.float64)
    B, n_tok, _ = x.shape
    assert n_tok == n_frames * cache.T
    c = x @ np.asarray(w_dkv, dtype=np.float64).T
    if use_rmsnorm:
        c = rmsnorm(c, gamma, eps)
    k = x @ np.asarray(w_kr, dtype=np.float64).T
    if spec is not None and k.shape[-1] > 0:
        k = rope3d(k, pos, spec)
    for n in range(n_tok):
        f = first_frame + n // cache.T
        s = sink_ring_slot(f, n % cache.T, cache.T, cache.W, cache.S)
        cache.c[:, s, :] = c[:, n, :]
        cache.kr[:, s, :] = k[:, n, :]
        cache.pos_of_slot[:, s, :] = np.asarray(pos)[:, n, :]
        cache.frame_of_slot[s] = f
    cache.frames_written = max(cache.frames_written, first_frame + n_frames)
    return c, k


# --------------------------------------------------------------------------
# Attention
# --------------------------------------------------------------------------
def softmax(s, axis=-1):
    """Plain softmax; subtracting the max does not change the value."""
    m = np.max(s, axis=axis, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=axis, keepdims=True)


def latent_attention(q_c, q_r, q_pos, keys_c, keys_k, head_dim, spec,
                     key_frames=None, query_last_frame=None, return_probs=False):
    """Absorbed-form attention of App. E for one batch element.

    q_c   : [Nq, H, d_c] absorbed content queries  A_h^T c^Q   (Eq. absorb-q)
    q_r   : [Nq, H, d_r] unrotated positional queries W_R,h^Q c^Q (Eq. qrope)
    q_pos : [Nq, 3]
    keys_c: [Nk, d_c] cached latents c^KV; keys_k: [Nk, d_r] rotated keys
    score = (q_c.c_j + RoPE3D(q_r).k_j) / sqrt(head_dim)   (Eq. score, R4)
    o_lat,h = sum_j p_hj c_j  (the latent output of Eq. absorb-v)
    Keys whose frame is after the query chunk's last frame are masked out
    (chunk-causal mask, App. D.4).
    """
    q_c = np.asarray(q_c, dtype=np.float64)
    q_r = np.asarray(q_r, dtype=np.float64)
    kc = np.asarray(keys_c, dtype=np.float64)
    kk = np.asarray(keys_k, dtype=np.float64)
    if q_r.shape[-1] > 0:
        q_rope = rope3d(q_r, np.asarray(q_pos)[:, None, :], spec)
    else:
        q_rope = q_r
    s = (np.einsum("nhc,jc->nhj", q_c, kc) + np.einsum("nhr,jr->nhj", q_rope, kk))
    s = s / math.sqrt(head_dim)
    if key_frames is not None and query_last_frame is not None:
        masked = np.asarray(key_frames) > query_last_frame
        s = np.where(masked[None, None, :], -np.inf, s)
    p = softmax(s, axis=-1)
    o = np.einsum("nhj,jc->nhc", p, kc)
    return (o, p) if return_probs else o


def window_attention(cache, b, q_c, q_r, q_pos, head_dim, spec):
    """Attention of a query chunk over the assembled window of a cache that
    stores k^R unrotated (App. D.4, D.5; readings R12, R13).

    cache : OracleCache filled by cache_append(..., spec=None)
    b     : batch element
    q_c, q_r : [Nq, H, d_c], [Nq, H, d_r] as for latent_attention
    q_pos : [Nq, 3] (t, h, w) with t the query token's absolute frame, which
            the window must hold
    Every held frame gets its window-local temporal coordinate; the cached
    keys and the queries are rotated at those coordinates, then the scores
    and outputs are those of latent_attention over the held slots.
    """
    slots = cache.valid_slots()
    fw = cache.frames_written
    key_pos = cache.pos_of_slot[b, slots].copy()
    key_pos[:, 0] = [window_local_time(cache.frame_of_slot[s], fw, cache.W, cache.S)
                     for s in slots]
    k_rope = rope3d(cache.kr[b, slots], key_pos, spec)
    q_local = np.array(q_pos, dtype=np.int64).copy()
    q_local[:, 0] = [window_local_time(t, fw, cache.W, cache.S) for t in q_local[:, 0]]
    return latent_attention(q_c, q_r, q_local, cache.c[b, slots], k_rope, head_dim, spec)


def reference_attention(x_q, pos_q, x_kv, pos_kv, w, head_dim, spec,
                        eps=1e-6, use_rmsnorm=True, key_frames=None,
                        query_last_frame=None, return_probs=False):
    """Non-absorbed training-time forward of Sec. 3.3 for one batch element.

    x_q [Nq, d], x_kv [Nk, d]; w is a dict of float64 weights:
      w_dkv [d_c, d], w_kr [d_r, d], w_dq [d_q, d],
      w_uk [H, d_nope, d_c], w_uv [H, d_v, d_c], w_uq [H, d_nope, d_q],
      w_qr [H, d_r, d_q]; optional gamma_kv [d_c], gamma_q [d_q], w_o [d, H*d_v].
    Returns the per-head outputs o [Nq, H, d_v] (and y = W_O o if w_o given).
    """
    x_q = np.asarray(x_q, dtype=np.float64)
    x_kv = np.asarray(x_kv, dtype=np.float64)
    # cache construction: Eq. ckv (+RMSNorm, App. D.2) and Eq. krope
    c_kv = x_kv @ w["w_dkv"].T
    if use_rmsnorm:
        c_kv = rmsnorm(c_kv, w.get("gamma_kv"), eps)
    k_R = x_kv @ w["w_kr"].T
    k_rope = rope3d(k_R, pos_kv, spec) if k_R.shape[-1] > 0 else k_R
    # Eq. reconstruct: per-head content keys and values from the shared latent
    k_nope = np.einsum("hec,jc->jhe", w["w_uk"], c_kv)
    v = np.einsum("hvc,jc->jhv", w["w_uv"], c_kv)
    # Eqs. cq, qnope, qrope
    c_q = x_q @ w["w_dq"].T
    if use_rmsnorm:
        c_q = rmsnorm(c_q, w.get("gamma_q"), eps)
    q_nope = np.einsum("heq,nq->nhe", w["w_uq"], c_q)
    q_R = np.einsum("hrq,nq->nhr", w["w_qr"], c_q)
    q_rope = rope3d(q_R, np.asarray(pos_q)[:, None, :], spec) if q_R.shape[-1] > 0 else q_R
    # Eq. score
    s = (np.einsum("nhe,jhe->nhj", q_nope, k_nope)
         + np.einsum("nhr,jr->nhj", q_rope, k_rope)) / math.sqrt(head_dim)
    if key_frames is not None and query_last_frame is not None:
        masked = np.asarray(key_frames) > query_last_frame
        s = np.where(masked[None, None, :], -np.inf, s)
    p = softmax(s, axis=-1)
    o = np.einsum("nhj,jhv->nhv", p, v)
    out = [o]
    if "w_o" in w:
        out.append(o.reshape(o.shape[0], -1) @ w["w_o"].T)
    if return_probs:
        out.append(p)
    return out[0] if len(out) == 1 else tuple(out)


def dense_attention(q, k, v, head_dim, return_probs=False):
    """Dense per-head attention, the layout VideoMLA replaces (App. C.1).

    q [Nq, H, d_h]; k, v [H, Nk, d_h] (RoPE already applied to q and k).
    o_h = softmax(q_h k_h^T / sqrt(head_dim)) v_h.
    """
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    s = np.einsum("nhd,hjd->nhj", q, k) / math.sqrt(head_dim)
    p = softmax(s, axis=-1)
    o = np.einsum("nhj,hjd->nhd", p, v)
    return (o, p) if return_probs else o


# --------------------------------------------------------------------------
# Absorption (App. E)
# --------------------------------------------------------------------------
def absorb_query(c_q, w_uq, w_uk):
    """q_c,h = A_h^T c^Q with A_h = (W_up,h^Q)^T W_up,h^K  (Eq. absorb-q)."""
    A = np.einsum("heq,hec->hqc", w_uq, w_uk)       # [H, d_q, d_c]
    return np.einsum("hqc,nq->nhc", A, np.asarray(c_q, dtype=np.float64))


def absorbed_query_matrices(w_uq, w_uk):
    """A_h = (W_up,h^Q)^T W_up,h^K in R^{d_q x d_c}, stacked over heads (App. E)."""
    return np.einsum("heq,hec->hqc", np.asarray(w_uq, dtype=np.float64),
                     np.asarray(w_uk, dtype=np.float64))


def absorbed_output_matrices(w_uv, w_o):
    """B_h = W_O,h W_up,h^V in R^{d x d_c}, stacked over heads (App. E)."""
    w_uv = np.asarray(w_uv, dtype=np.float64)
    w_o = np.asarray(w_o, dtype=np.float64)
    H, d_v, _ = w_uv.shape
    return np.stack([w_o[:, h * d_v:(h + 1) * d_v] @ w_uv[h] for h in range(H)])


def per_head_output_from_latent(o_lat, w_uv):
    """o_h = W_up,h^V o_lat,h : the value up-projection applied after the sum."""
    return np.einsum("hvc,nhc->nhv", w_uv, np.asarray(o_lat, dtype=np.float64))


def absorb_output(o_lat, w_uv, w_o):
    """y = sum_h B_h o_lat,h with B_h = W_O,h W_up,h^V  (Eq. absorb-v)."""
    H, d_v, _ = w_uv.shape
    Bh = np.stack([w_o[:, h * d_v:(h + 1) * d_v] @ w_uv[h] for h in range(H)])
    return np.einsum("hdc,nhc->nd", Bh, np.asarray(o_lat, dtype=np.float64))


# --------------------------------------------------------------------------
# Cost model (Sec. 3.1; Table 1; App. E)
# --------------------------------------------------------------------------
def cache_scalars_per_token(d_c, d_r):
    """Latent cache: d_c + d_rope scalars per token per layer."""
    return d_c + d_r


def dense_scalars_per_token(n_h, d_h):
    """Dense per-head KV: 2 n_h d_h scalars per token per layer."""
    return 2 * n_h * d_h


def latent_attention_flops(rows, keys, d_c, d_r):
    """Multiply-adds x2 of the absorbed form: QK^T over d_c+d_r, PV over d_c."""
    return 2.0 * rows * keys * (d_c + d_r) + 2.0 * rows * keys * d_c

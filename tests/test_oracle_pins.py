"""Pins for the float64 oracle: each test checks it against something other
than itself -- numbers the paper prints, closed forms, textbook or library
routines, invariants, and brute force on tiny inputs."""

import math
import os
from collections import deque

import numpy as np
import pytest
import torch

from oracle import mla_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                k, v = line.split("=")
                vals[k.strip()] = float(v)
    return vals


def _rng(seed=0):
    return np.random.default_rng(seed)


def _sdpa(q, k, v, scale=None):
    """torch's scaled_dot_product_attention in float64 (the library routine)."""
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))
    return torch.nn.functional.scaled_dot_product_attention(
        t(q), t(k), t(v), scale=scale).numpy()


# ---------------------------------------------------------------- cache sizes
def test_cache_sizes_match_paper():
    g = _golden("paper_cache_sizes.txt")
    lat = O.cache_scalars_per_token(192, 32)
    dense = O.dense_scalars_per_token(12, 128)
    assert lat == g["latent_scalars_per_token"]
    assert dense == g["dense_scalars_per_token"]
    assert round(100 * (1 - lat / dense), 1) == g["reduction_percent"]
    assert round(dense / lat, 1) == g["reduction_factor"]
    scalars = 21 * 1560 * 30 * dense
    assert round(scalars / 1e9, 2) == g["dense_cache_scalars_billions"]
    assert round(scalars * 2 / 1e9, 1) == g["dense_cache_gb_bf16"]
    frac = 1 - g["scd_cached_layers"] / g["scd_total_layers"]
    assert round(100 * frac, 1) == g["scd_reduction_percent"]
    scd = dense * g["scd_cached_layers"] / (lat * g["scd_total_layers"])
    assert round(scd, 1) == g["scd_vs_videomla_factor"]
    for dc in (64, 128, 256, 512):
        ratio = dense / O.cache_scalars_per_token(dc, 32)
        assert round(ratio, 2) == g[f"mem_ratio_dc{dc}"], dc


# ---------------------------------------------------------------------- RoPE
def test_rope_single_axis_is_complex_rotation():
    """Restricted to one axis, 3D-RoPE is z -> z * exp(i pos w) (textbook)."""
    spec = O.RopeSpec(pairs=(5, 0, 0), axis_dims=(10, 2, 2), theta=10000.0)
    rng = _rng(1)
    v = rng.standard_normal((7, 10))
    pos = np.zeros((7, 3), dtype=np.int64)
    pos[:, 0] = rng.integers(0, 1000, 7)
    out = O.rope3d(v, pos, spec)
    z = v[:, 0::2] + 1j * v[:, 1::2]
    w = 10000.0 ** (-np.arange(5) * 2.0 / 10)
    zr = z * np.exp(1j * pos[:, :1] * w[None, :])
    np.testing.assert_allclose(out[:, 0::2], zr.real, rtol=0, atol=1e-12)
    np.testing.assert_allclose(out[:, 1::2], zr.imag, rtol=0, atol=1e-12)


def test_rope_structure():
    spec = O.RopeSpec(pairs=(6, 5, 5), axis_dims=(44, 42, 42))
    inv, axis = O.rope_inv_freq(spec)
    assert len(inv) == 16 and spec.d_r == 32
    assert list(axis) == [0] * 6 + [1] * 5 + [2] * 5
    for a in range(3):                       # highest band first, decreasing
        f = inv[axis == a]
        assert f[0] == 1.0 and np.all(np.diff(f) < 0)
    rng = _rng(2)
    v = rng.standard_normal((5, 32))
    # position zero is the identity; rotation preserves every pair's norm
    np.testing.assert_array_equal(O.rope3d(v, np.zeros((5, 3), int), spec), v)
    pos = rng.integers(0, 1024, (5, 3))
    r = O.rope3d(v, pos, spec)
    np.testing.assert_allclose(r[:, 0::2] ** 2 + r[:, 1::2] ** 2,
                               v[:, 0::2] ** 2 + v[:, 1::2] ** 2, rtol=1e-12)


def test_rope_relative_position():
    """<R(p) q, R(p') k> depends only on p - p' (what makes rotate-at-append
    equal to window-relative re-indexing, Sec. 3.2 / App. D.5)."""
    spec = O.RopeSpec(pairs=(4, 6, 6))
    rng = _rng(3)
    q, k = rng.standard_normal((2, 32))
    p1, p2 = np.array([17, 3, 40]), np.array([5, 29, 2])
    base = O.rope3d(q, p1, spec) @ O.rope3d(k, p2, spec)
    for shift in ([900, 0, 0], [1, 2, 3], [0, 17, 0]):
        s = np.array(shift)
        got = O.rope3d(q, p1 + s, spec) @ O.rope3d(k, p2 + s, spec)
        assert abs(got - base) < 1e-9
    # and it does change with the difference
    got = O.rope3d(q, p1 + np.array([1, 0, 0]), spec) @ O.rope3d(k, p2, spec)
    assert abs(got - base) > 1e-6


# ------------------------------------------------------------------- RMSNorm
def test_rmsnorm_matches_torch_and_invariants():
    rng = _rng(4)
    v = rng.standard_normal((6, 192)) * 3.0
    g = rng.standard_normal(192)
    ref = torch.nn.functional.rms_norm(torch.from_numpy(v), (192,),
                                       torch.from_numpy(g), eps=1e-6).numpy()
    np.testing.assert_allclose(O.rmsnorm(v, g, 1e-6), ref, rtol=1e-12, atol=1e-12)
    u = O.rmsnorm(v, None, 0.0)
    np.testing.assert_allclose(np.mean(u * u, axis=-1), 1.0, rtol=1e-12)
    np.testing.assert_allclose(O.rmsnorm(7.5 * v, None, 0.0), u, rtol=1e-12)


# ---------------------------------------------------------------- ring / FIFO
@pytest.mark.parametrize("schedule", [
    [(0, 1), (1, 1), (2, 1), (3, 1), (4, 1), (5, 1), (6, 1)],
    [(0, 3), (3, 3), (3, 3), (6, 3), (9, 3), (12, 3), (12, 3), (15, 3)],
    [(0, 2), (2, 2), (4, 1), (5, 3), (8, 4)],
])
def test_ring_is_fifo(schedule):
    """Simulate the window as a FIFO queue of frames and compare slot contents."""
    T, W = 3, 4
    cache = O.OracleCache(1, T, W, d_c=2, d_r=0)
    q = deque()
    for first, n in schedule:
        x = np.zeros((1, n * T, 4))
        for i in range(n * T):                         # token carries its identity
            x[0, i, 0] = first + i // T
            x[0, i, 1] = i % T
        w_dkv = np.eye(2, 4)
        O.cache_append(cache, x, w_dkv, np.zeros((0, 4)), np.zeros((1, n * T, 3), int),
                       first, n, use_rmsnorm=False)
        for f in range(first, first + n):
            if f not in q:
                q.append(f)
            while len(q) > W:
                q.popleft()
        held = sorted(q)
        assert O.window_frames(cache.frames_written, W) == held
        valid = cache.valid_slots()
        assert len(valid) == len(held) * T
        for s in valid:                               # slot holds its frame's tokens
            assert cache.c[0, s, 0] == cache.frame_of_slot[s]
            assert cache.c[0, s, 1] == s % T
        assert sorted(set(cache.frame_of_slot[valid])) == held


# ------------------------------------------------------------- attention pins
def _small_weights(rng, d, H, dh, dc, dr, dq):
    dn = dh - dr
    n = lambda *s: rng.standard_normal(s) * s[-1] ** -0.5
    return {"w_dkv": n(dc, d), "w_kr": n(dr, d), "w_dq": n(dq, d),
            "w_uk": n(H, dn, dc), "w_uv": n(H, dh, dc), "w_uq": n(H, dn, dq),
            "w_qr": n(H, dr, dq), "w_o": n(d, H * dh),
            "gamma_kv": 1 + 0.1 * rng.standard_normal(dc),
            "gamma_q": 1 + 0.1 * rng.standard_normal(dq)}


def test_dense_reduction_identity_projections():
    """d_r = 0, d_c = n_h d_h, identity down-projections and head-selector
    up-projections: MLA reduces to textbook MHA with Q = K = V = x."""
    rng = _rng(5)
    H, dh = 3, 4
    d = H * dh
    sel = np.stack([np.eye(d)[h * dh:(h + 1) * dh] for h in range(H)])   # [H, dh, d]
    w = {"w_dkv": np.eye(d), "w_kr": np.zeros((0, d)), "w_dq": np.eye(d),
         "w_uk": sel, "w_uv": sel, "w_uq": sel, "w_qr": np.zeros((H, 0, d))}
    spec = O.RopeSpec(pairs=(0, 0, 0))
    xq, xkv = rng.standard_normal((5, d)), rng.standard_normal((9, d))
    o = O.reference_attention(xq, np.zeros((5, 3), int), xkv, np.zeros((9, 3), int),
                              w, dh, spec, use_rmsnorm=False)
    qh = xq.reshape(5, H, dh).transpose(1, 0, 2)
    kh = xkv.reshape(9, H, dh).transpose(1, 0, 2)
    ref = _sdpa(qh, kh, kh).transpose(1, 0, 2)
    np.testing.assert_allclose(o, ref, rtol=1e-12, atol=1e-12)


def test_dense_reduction_joint_kv():
    """d_c = 2 n_h d_h with W_dn^KV = [W_K; W_V]: MLA is dense MHA with
    independent keys and values."""
    rng = _rng(6)
    H, dh = 2, 4
    d = H * dh
    WQ, WK, WV = rng.standard_normal((3, d, d))
    selK = np.stack([np.eye(2 * d)[h * dh:(h + 1) * dh] for h in range(H)])
    selV = np.stack([np.eye(2 * d)[d + h * dh:d + (h + 1) * dh] for h in range(H)])
    selQ = np.stack([np.eye(d)[h * dh:(h + 1) * dh] for h in range(H)])
    w = {"w_dkv": np.concatenate([WK, WV]), "w_kr": np.zeros((0, d)), "w_dq": WQ,
         "w_uk": selK, "w_uv": selV, "w_uq": selQ, "w_qr": np.zeros((H, 0, d))}
    xq, xkv = rng.standard_normal((4, d)), rng.standard_normal((6, d))
    o = O.reference_attention(xq, np.zeros((4, 3), int), xkv, np.zeros((6, 3), int),
                              w, dh, O.RopeSpec(pairs=(0, 0, 0)), use_rmsnorm=False)
    split = lambda a: a.reshape(a.shape[0], H, dh).transpose(1, 0, 2)
    ref = _sdpa(split(xq @ WQ.T), split(xkv @ WK.T), split(xkv @ WV.T))
    np.testing.assert_allclose(o, ref.transpose(1, 0, 2), rtol=1e-11, atol=1e-11)


def test_latent_attention_is_sdpa_over_concatenated_keys():
    """The absorbed form is one SDPA with queries [q_c, RoPE(q_r)], keys
    [c, k] and values c, scaled by 1/sqrt(d_h) (Eq. score, App. E)."""
    rng = _rng(7)
    spec = O.RopeSpec(pairs=(2, 1, 1))
    Nq, H, dc, dr, Nk, dh = 5, 3, 6, 8, 11, 16
    qc, qr = rng.standard_normal((Nq, H, dc)), rng.standard_normal((Nq, H, dr))
    qpos = rng.integers(0, 50, (Nq, 3))
    kc, kk = rng.standard_normal((Nk, dc)), rng.standard_normal((Nk, dr))
    o, p = O.latent_attention(qc, qr, qpos, kc, kk, dh, spec, return_probs=True)
    np.testing.assert_allclose(p.sum(-1), 1.0, rtol=0, atol=1e-12)
    # rotate each head's q_r by hand via complex multiplication
    inv, axis = O.rope_inv_freq(spec)
    z = qr[..., 0::2] + 1j * qr[..., 1::2]
    ang = qpos[:, None, axis] * inv[None, None, :]
    zr = z * np.exp(1j * ang)
    qrot = np.empty_like(qr)
    qrot[..., 0::2], qrot[..., 1::2] = zr.real, zr.imag
    q = np.concatenate([qc, qrot], -1).transpose(1, 0, 2)
    k = np.concatenate([kc, kk], -1)[None].repeat(H, 0)
    v = kc[None].repeat(H, 0)
    ref = _sdpa(q, k, v, scale=1 / math.sqrt(dh)).transpose(1, 0, 2)
    np.testing.assert_allclose(o, ref, rtol=1e-12, atol=1e-12)


def _layer_setup(seed, T=4, W=3, chunk=2, n_chunks=3, pairs=(2, 1, 1)):
    rng = _rng(seed)
    d, H, dh, dc, dq = 16, 2, 8, 6, 10
    spec = O.RopeSpec(pairs=pairs, axis_dims=(8, 6, 6))
    dr = spec.d_r
    w = _small_weights(rng, d, H, dh, dc, dr, dq)
    cache = O.OracleCache(1, T, W, dc, dr)
    xs, ps = [], []
    for c in range(n_chunks):
        first = c * chunk
        x = rng.standard_normal((1, chunk * T, d))
        pos = np.stack([np.repeat(np.arange(first, first + chunk), T),
                        np.tile(np.arange(T) // 2, chunk), np.tile(np.arange(T) % 2, chunk)],
                       -1)[None]
        O.cache_append(cache, x, w["w_dkv"], w["w_kr"], pos, first, chunk,
                       gamma=w["gamma_kv"], spec=spec)
        xs.append(x[0])
        ps.append(pos[0])
    return rng, w, spec, cache, xs, ps, (d, H, dh, dc, dr, dq)


def test_absorption_identity():
    """Absorbed inference form equals the non-absorbed training form (App. E)."""
    rng, w, spec, cache, xs, ps, (d, H, dh, dc, dr, dq) = _layer_setup(8)
    valid = cache.valid_slots()
    # window tokens in slot order, with their inputs and positions
    T, W = cache.T, cache.W
    held = O.window_frames(cache.frames_written, W)
    allx = np.concatenate(xs)
    allp = np.concatenate(ps)
    first_frame_of = {f: i for i, f in enumerate(range(len(allx) // T))}
    tok = [first_frame_of[cache.frame_of_slot[s]] * T + s % T for s in valid]
    x_kv, pos_kv = allx[tok], allp[tok]
    assert sorted(set(pos_kv[:, 0])) == held
    x_q, pos_q = xs[-1], ps[-1]
    o_ref, y_ref = O.reference_attention(x_q, pos_q, x_kv, pos_kv, w, dh, spec)
    c_q = O.rmsnorm(x_q @ w["w_dq"].T, w["gamma_q"])
    q_c = O.absorb_query(c_q, w["w_uq"], w["w_uk"])
    q_r = np.einsum("hrq,nq->nhr", w["w_qr"], c_q)
    o_lat = O.latent_attention(q_c, q_r, pos_q, cache.c[0, valid], cache.kr[0, valid],
                               dh, spec)
    np.testing.assert_allclose(O.per_head_output_from_latent(o_lat, w["w_uv"]), o_ref,
                               rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(O.absorb_output(o_lat, w["w_uv"], w["w_o"]), y_ref,
                               rtol=1e-10, atol=1e-12)


def test_shift_invariance():
    """A common offset added to every position leaves the output unchanged."""
    outs = []
    for shift in ([0, 0, 0], [700, 5, 11]):
        rng = _rng(9)
        spec = O.RopeSpec(pairs=(2, 1, 1), axis_dims=(8, 6, 6))
        kc, kr = rng.standard_normal((12, 6)), rng.standard_normal((12, 8))
        kpos = rng.integers(0, 40, (12, 3)) + np.array(shift)
        kk = O.rope3d(kr, kpos, spec)
        qc, qr = rng.standard_normal((3, 2, 6)), rng.standard_normal((3, 2, 8))
        qpos = rng.integers(0, 40, (3, 3)) + np.array(shift)
        outs.append(O.latent_attention(qc, qr, qpos, kc, kk, 8, spec))
    np.testing.assert_allclose(outs[1], outs[0], rtol=0, atol=1e-9)


def test_chunk_causal_mask_drops_later_frames():
    """Keys of frames after the query chunk are invisible (App. D.4): masking
    them equals attending over the earlier keys only."""
    rng = _rng(10)
    spec = O.RopeSpec(pairs=(1, 1, 1), axis_dims=(6, 6, 6))
    kc, kk = rng.standard_normal((10, 4)), rng.standard_normal((10, 6))
    frames = np.array([0, 0, 1, 1, 2, 2, 3, 3, 4, 4])
    qc, qr = rng.standard_normal((2, 3, 4)), rng.standard_normal((2, 3, 6))
    qpos = np.array([[2, 0, 0], [2, 1, 0]])
    o = O.latent_attention(qc, qr, qpos, kc, kk, 8, spec, key_frames=frames,
                           query_last_frame=2)
    keep = frames <= 2
    o2 = O.latent_attention(qc, qr, qpos, kc[keep], kk[keep], 8, spec)
    np.testing.assert_allclose(o, o2, rtol=1e-13, atol=1e-13)


def test_hand_case_two_tokens():
    """One head, d_nope = 2, d_rope = 2 (one temporal pair, frequency 1),
    two cached tokens at t = 0 and t = 1, query at t = 1. Closed form:
    s_j = (q_n . k_n,j + q_r . R(t_q - t_j) k_j) / 2, o = sum softmax(s)_j v_j."""
    spec = O.RopeSpec(pairs=(1, 0, 0), axis_dims=(2, 2, 2))
    # latent c_j = (1, 0) and (0, 2); W_up^K = I, W_up^V = [[1, 1], [0, 3]] (d_v = 2)
    c = np.array([[1.0, 0.0], [0.0, 2.0]])
    kR = np.array([[1.0, 0.0], [0.0, 1.0]])
    pos_k = np.array([[0, 0, 0], [1, 0, 0]])
    qn = np.array([1.0, 1.0])
    qR = np.array([1.0, 0.0])
    pos_q = np.array([[1, 0, 0]])
    w_uv = np.array([[[1.0, 1.0], [0.0, 3.0]]])
    k_rope = O.rope3d(kR, pos_k, spec)
    # q_c = W_up^K^T q_n = q_n with W_up^K = I
    o_lat = O.latent_attention(qn[None, None, :], qR[None, None, :], pos_q, c, k_rope, 4, spec)
    o = O.per_head_output_from_latent(o_lat, w_uv)[0, 0]
    # by hand: R(1) q_R = (cos1, sin1); k_rope_0 = (1,0); k_rope_1 = R(1)(0,1) = (-sin1, cos1)
    s0 = (1.0 + math.cos(1.0)) / 2.0
    s1 = (2.0 + (-math.cos(1.0) * math.sin(1.0) + math.sin(1.0) * math.cos(1.0))) / 2.0
    p0 = math.exp(s0) / (math.exp(s0) + math.exp(s1))
    p1 = 1.0 - p0
    v0, v1 = np.array([1.0, 0.0]), np.array([2.0, 6.0])       # W_up^V c_j
    np.testing.assert_allclose(o, p0 * v0 + p1 * v1, rtol=0, atol=1e-14)


def test_brute_force_loops():
    """Pure-Python loops over the non-absorbed definition on a tiny layer."""
    rng, w, spec, cache, xs, ps, (d, H, dh, dc, dr, dq) = _layer_setup(11, n_chunks=2)
    x_q, pos_q = xs[-1], ps[-1]
    x_kv = np.concatenate(xs)
    pos_kv = np.concatenate(ps)
    o, _y = O.reference_attention(x_q, pos_q, x_kv, pos_kv, w, dh, spec)
    inv, axis = O.rope_inv_freq(spec)
    dn = dh - dr

    def mv(M, v):
        return [sum(M[i][j] * v[j] for j in range(len(v))) for i in range(len(M))]

    def rms(v, g):
        r = math.sqrt(sum(a * a for a in v) / len(v) + 1e-6)
        return [v[i] / r * g[i] for i in range(len(v))]

    def rot(v, p):
        out = list(v)
        for i in range(len(inv)):
            a = p[axis[i]] * inv[i]
            out[2 * i] = v[2 * i] * math.cos(a) - v[2 * i + 1] * math.sin(a)
            out[2 * i + 1] = v[2 * i] * math.sin(a) + v[2 * i + 1] * math.cos(a)
        return out

    for n in range(len(x_q)):
        cq = rms(mv(w["w_dq"], x_q[n]), w["gamma_q"])
        for h in range(H):
            qn = mv(w["w_uq"][h], cq)
            qr = rot(mv(w["w_qr"][h], cq), pos_q[n])
            scores = []
            vals = []
            for j in range(len(x_kv)):
                ckv = rms(mv(w["w_dkv"], x_kv[j]), w["gamma_kv"])
                kn = mv(w["w_uk"][h], ckv)
                kr = rot(mv(w["w_kr"], x_kv[j]), pos_kv[j])
                s = (sum(qn[i] * kn[i] for i in range(dn))
                     + sum(qr[i] * kr[i] for i in range(dr))) / math.sqrt(dh)
                scores.append(s)
                vals.append(mv(w["w_uv"][h], ckv))
            m = max(scores)
            e = [math.exp(s - m) for s in scores]
            z = sum(e)
            ref = [sum(e[j] * vals[j][i] for j in range(len(e))) / z for i in range(dh)]
            np.testing.assert_allclose(o[n, h], ref, rtol=1e-11, atol=1e-12)


def test_absorbed_matrices_apply_like_the_absorbed_maps():
    """A_h and B_h applied as matrices equal absorb_query / absorb_output, and
    B_h o_lat,h equals W_O,h (W_up,h^V o_lat,h) -- the two groupings of Eq. absorb-v."""
    rng = _rng(12)
    H, dn, dq, dc, dh, d = 3, 4, 6, 5, 7, 9
    w_uq, w_uk = rng.standard_normal((H, dn, dq)), rng.standard_normal((H, dn, dc))
    w_uv, w_o = rng.standard_normal((H, dh, dc)), rng.standard_normal((d, H * dh))
    c_q = rng.standard_normal((4, dq))
    A = O.absorbed_query_matrices(w_uq, w_uk)
    np.testing.assert_allclose(np.einsum("hqc,nq->nhc", A, c_q), O.absorb_query(c_q, w_uq, w_uk),
                               rtol=1e-12, atol=1e-12)
    o_lat = rng.standard_normal((4, H, dc))
    B = O.absorbed_output_matrices(w_uv, w_o)
    y = np.einsum("hdc,nhc->nd", B, o_lat)
    o_h = O.per_head_output_from_latent(o_lat, w_uv)
    np.testing.assert_allclose(y, o_h.reshape(4, -1) @ w_o.T, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(O.absorb_output(o_lat, w_uv, w_o), y, rtol=1e-12, atol=1e-12)


def test_dense_attention_is_sdpa():
    """The dense baseline is torch's SDPA per head."""
    rng = _rng(13)
    q, k, v = rng.standard_normal((6, 3, 8)), rng.standard_normal((3, 10, 8)), rng.standard_normal((3, 10, 8))
    ref = _sdpa(q.transpose(1, 0, 2), k, v).transpose(1, 0, 2)
    np.testing.assert_allclose(O.dense_attention(q, k, v, 8), ref, rtol=1e-12, atol=1e-12)


def test_flop_count_matches_numpy_contraction_count():
    """latent_attention_flops against NumPy's own operation count of the three
    contractions latent_attention performs (scores over c and over k, then
    P times c): two FLOPs per multiply-add of each einsum."""
    import re

    def naive(spec, *shapes):
        info = np.einsum_path(spec, *[np.zeros(s) for s in shapes], optimize="greedy")[1]
        return float(re.search(r"Naive FLOP count:\s*([0-9.e+]+)", info).group(1))

    for nq, H, nk, dc, dr in [(3, 2, 7, 5, 4), (4, 3, 11, 8, 2), (2, 1, 1, 6, 0)]:
        got = O.latent_attention_flops(nq * H, nk, dc, dr)
        want = naive("nhc,jc->nhj", (nq, H, dc), (nk, dc)) + naive("nhj,jc->nhc", (nq, H, nk), (nk, dc))
        if dr:
            want += naive("nhr,jr->nhj", (nq, H, dr), (nk, dr))
        assert got == want, (got, want)

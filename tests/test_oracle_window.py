"""Pins of the oracle's long-rollout cache (App. D.4: one sink frame plus a
FIFO window of the newest frames) and of window-relative RoPE re-indexing
(App. D.5: k^R cached unrotated, keys and queries rotated at window-local
temporal coordinates when the window is assembled).

The pins are independent of the code they check: a list model of the sink +
FIFO window, and RoPE's relative-position property (scores depend only on
position differences), which makes re-indexed attention equal to attention
with absolute positions after a known relabelling of the frames."""

import numpy as np
import pytest

from oracle import mla_oracle as O

SPEC = O.RopeSpec(pairs=(2, 1, 1), axis_dims=(8, 6, 6))


def _identity_append(cache, first, n):
    """Append n frames whose tokens carry (frame, k) in c."""
    T = cache.T
    x = np.zeros((1, n * T, 4))
    for i in range(n * T):
        x[0, i, 0] = first + i // T
        x[0, i, 1] = i % T
    O.cache_append(cache, x, np.eye(2, 4), np.zeros((0, 4)), np.zeros((1, n * T, 3), int),
                   first, n, use_rmsnorm=False)


@pytest.mark.parametrize("sink", [0, 1, 2])
@pytest.mark.parametrize("schedule", [
    [(f, 1) for f in range(15)],
    [(0, 3), (3, 3), (3, 3), (6, 3), (9, 3), (12, 3), (12, 3), (15, 3), (18, 3)],
    [(0, 2), (2, 2), (4, 1), (5, 3), (8, 2), (10, 1)],
])
def test_sink_window_is_sinks_plus_fifo(schedule, sink):
    """List model: the first `sink` frames are never evicted; later frames go
    through a FIFO queue of W - sink frames; slots hold their frame's tokens."""
    T, W = 3, 5
    cache = O.OracleCache(1, T, W, d_c=2, d_r=0, sink_frames=sink)
    sinks, fifo = [], []
    for first, n in schedule:
        _identity_append(cache, first, n)
        for f in range(first, first + n):
            if f < sink:
                if f not in sinks:
                    sinks.append(f)
            elif f not in fifo:
                fifo.append(f)
                if len(fifo) > W - sink:
                    fifo.pop(0)
        held = sorted(sinks) + fifo
        assert cache.held_frames() == held
        valid = cache.valid_slots()
        assert len(valid) == len(held) * T
        for s in valid:
            assert cache.c[0, s, 0] == cache.frame_of_slot[s]
            assert cache.c[0, s, 1] == s % T
        # before the first eviction the window fills the slots in order
        if cache.frames_written <= W:
            assert list(valid) == list(range(cache.frames_written * T))


def test_sink_zero_is_the_plain_ring():
    for f in range(40):
        for k in range(3):
            assert O.sink_ring_slot(f, k, 3, 7, 0) == O.ring_slot(f, k, 3, 7)
    for fw in range(30):
        assert O.sink_window_frames(fw, 7, 0) == O.window_frames(fw, 7)


def test_local_time_numbers_the_held_frames():
    W, S = 7, 1
    for fw in range(1, 40):
        held = O.sink_window_frames(fw, W, S)
        local = [O.window_local_time(f, fw, W, S) for f in held]
        assert local == list(range(len(held)))
        if fw <= W:                                       # nothing evicted yet
            assert held == list(range(fw))
    with pytest.raises(ValueError):
        O.window_local_time(3, 20, W, S)                  # evicted long ago


def _rollout(seed, W, S, frames, chunk=3, T=4, dc=6):
    """Append `frames` frames in chunks to two caches: one storing k^R
    unrotated (the window path) and one rotating at append with absolute
    positions. Returns both caches and a query chunk of the newest frames."""
    rng = np.random.default_rng(seed)
    d = 10
    w_dkv = rng.standard_normal((dc, d))
    w_kr = rng.standard_normal((SPEC.d_r, d))
    raw = O.OracleCache(1, T, W, dc, SPEC.d_r, sink_frames=S)
    rot = O.OracleCache(1, T, W, dc, SPEC.d_r, sink_frames=S)
    hw = np.stack([np.arange(T) // 2, np.arange(T) % 2], -1)
    for first in range(0, frames, chunk):
        n = min(chunk, frames - first)
        x = rng.standard_normal((1, n * T, d))
        pos = np.concatenate([np.repeat(np.arange(first, first + n), T)[:, None],
                              np.tile(hw, (n, 1))], -1)[None]
        O.cache_append(raw, x, w_dkv, w_kr, pos, first, n)
        O.cache_append(rot, x, w_dkv, w_kr, pos, first, n, spec=SPEC)
    last = frames - 1
    q_frames = np.arange(last - chunk + 1, last + 1)
    q_pos = np.concatenate([np.repeat(q_frames, T)[:, None], np.tile(hw, (chunk, 1))], -1)
    q_c = rng.standard_normal((len(q_pos), 2, dc))
    q_r = rng.standard_normal((len(q_pos), 2, SPEC.d_r))
    return raw, rot, q_c, q_r, q_pos


@pytest.mark.parametrize("frames", [3, 6, 9, 15, 24])
def test_contiguous_window_reindexing_equals_absolute_rotation(frames):
    """No sink: the window is contiguous, so local coordinates differ from the
    absolute ones by one shift and the re-indexed attention equals the
    rotate-at-append attention at absolute positions (RoPE relativity)."""
    raw, rot, q_c, q_r, q_pos = _rollout(3, W=6, S=0, frames=frames)
    got = O.window_attention(raw, 0, q_c, q_r, q_pos, 8, SPEC)
    valid = rot.valid_slots()
    ref = O.latent_attention(q_c, q_r, q_pos, rot.c[0, valid], rot.kr[0, valid], 8, SPEC)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-10)


@pytest.mark.parametrize("frames", [9, 12, 21, 30])
def test_sink_reindexing_moves_the_sink_next_to_the_window(frames):
    """One sink frame, window W = 7: once frames were evicted the sink's local
    time is 0 and the local frames follow at 1..6, which by RoPE relativity is
    the absolute-position attention with the sink relabelled as the frame
    right before the oldest local frame."""
    W, S = 7, 1
    raw, _rot, q_c, q_r, q_pos = _rollout(5, W=W, S=S, frames=frames)
    valid = raw.valid_slots()
    oldest_local = frames - (W - S)
    kpos = raw.pos_of_slot[0, valid].copy()
    kpos[raw.frame_of_slot[valid] == 0, 0] = oldest_local - 1
    k_abs = O.rope3d(raw.kr[0, valid], kpos, SPEC)
    ref = O.latent_attention(q_c, q_r, q_pos, raw.c[0, valid], k_abs, 8, SPEC)
    got = O.window_attention(raw, 0, q_c, q_r, q_pos, 8, SPEC)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-10)
    # and the relabelling matters: the sink left at absolute time 0 differs
    k_far = O.rope3d(raw.kr[0, valid], raw.pos_of_slot[0, valid], SPEC)
    far = O.latent_attention(q_c, q_r, q_pos, raw.c[0, valid], k_far, 8, SPEC)
    assert np.max(np.abs(far - got)) > 1e-6


def test_sink_window_before_eviction_is_absolute():
    """Up to W frames nothing is evicted and local time is absolute time."""
    raw, rot, q_c, q_r, q_pos = _rollout(7, W=7, S=1, frames=6)
    valid = rot.valid_slots()
    ref = O.latent_attention(q_c, q_r, q_pos, rot.c[0, valid], rot.kr[0, valid], 8, SPEC)
    np.testing.assert_allclose(O.window_attention(raw, 0, q_c, q_r, q_pos, 8, SPEC), ref,
                               rtol=0, atol=1e-12)


def test_window_attention_matches_brute_force_loops():
    """Pure-Python loops, independent of the oracle's vectorised code: the held
    frames are numbered by hand, every pair is rotated with explicit cos/sin at
    (local t, h, w), and the softmax is summed term by term."""
    import math
    spec = O.RopeSpec(pairs=(2, 1, 0), axis_dims=(4, 2, 2), theta=10000.0)
    T, W, S, dc, d = 2, 3, 1, 2, 5
    rng = np.random.default_rng(11)
    cache = O.OracleCache(1, T, W, dc, spec.d_r, sink_frames=S)
    w_dkv = rng.standard_normal((dc, d))
    w_kr = rng.standard_normal((spec.d_r, d))
    for f in range(6):
        x = rng.standard_normal((1, T, d))
        pos = np.array([[[f, k, 0] for k in range(T)]])
        O.cache_append(cache, x, w_dkv, w_kr, pos, f, 1)
    q_c = rng.standard_normal((3, 1, dc))
    q_r = rng.standard_normal((3, 1, spec.d_r))
    q_pos = np.array([[5, 0, 0], [5, 1, 0], [4, 1, 0]])
    got = O.window_attention(cache, 0, q_c, q_r, q_pos, 4, spec)

    held = [0, 4, 5]                         # the sink, then the two newest frames
    local = {f: i for i, f in enumerate(held)}
    bands = [(0, 0), (0, 1), (1, 0)]         # (axis, index within the axis) per pair

    def rotate(v, pos):
        out = []
        for p, (a, i) in enumerate(bands):
            ang = pos[a] * spec.theta ** (-2.0 * i / spec.axis_dims[a])
            x0, x1 = v[2 * p], v[2 * p + 1]
            out += [x0 * math.cos(ang) - x1 * math.sin(ang), x0 * math.sin(ang) + x1 * math.cos(ang)]
        return out

    keys = []
    for s in range(W * T):
        f = int(cache.frame_of_slot[s])
        if f in local:
            h = int(cache.pos_of_slot[0, s, 1])
            keys.append((list(cache.c[0, s]), rotate(list(cache.kr[0, s]), (local[f], h, 0))))
    assert len(keys) == 3 * T
    for n in range(3):
        qr = rotate(list(q_r[n, 0]), (local[int(q_pos[n, 0])], int(q_pos[n, 1]), 0))
        scores = [(sum(q_c[n, 0, i] * c[i] for i in range(dc)) +
                   sum(qr[i] * k[i] for i in range(spec.d_r))) / 2.0 for c, k in keys]
        mx = max(scores)
        e = [math.exp(sc - mx) for sc in scores]
        z = sum(e)
        o = [sum(e[j] / z * keys[j][0][i] for j in range(len(keys))) for i in range(dc)]
        np.testing.assert_allclose(got[n, 0], o, rtol=0, atol=1e-12)

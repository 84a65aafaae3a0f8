"""GPU parity of the long-rollout cache (App. D.4: sink frames kept for good,
the newest frames in FIFO order) and of window-relative RoPE (App. D.5: k^R
cached unrotated, keys and queries rotated at window-local times when the
window is assembled), through the C ABI, against the float64 oracle."""

import numpy as np
import pytest
import torch

from oracle import mla_oracle as O
from paper_2605_30351_gb300 import synth
from paper_2605_30351_gb300 import videomla as V

from test_gpu_parity import assert_close, f64, spec_of

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    V.load()
    V.mla_device_status(clear=True)
    yield
    assert V.mla_device_status(clear=True) == V.MLA_OK


def window_chunks(w, weights, chunks, flags=0, seed=700):
    """Append chunks to a rotate-at-use cache on the GPU and in the oracle."""
    cfg = V.make_config(w, flags | V.MLA_FLAG_ROTATE_AT_USE)
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    oc = O.OracleCache(w.batch, w.tokens_per_frame, w.window_frames, w.d_c, w.d_r,
                       sink_frames=w.sink_frames)
    dev = {k: v.cuda() for k, v in weights.items()}
    for i, (first, n) in enumerate(chunks):
        x = synth.draw_tokens(w, n * w.tokens_per_frame, seed + i)
        pos = synth.grid_positions(w, first, n)
        V.mla_cache_append(cache, x.cuda(), dev["w_dkv"], dev["gamma_kv"], dev["w_kr"], None,
                           first, n)
        O.cache_append(oc, f64(x), f64(weights["w_dkv"]), f64(weights["w_kr"]), pos.numpy(),
                       first, n, gamma=f64(weights["gamma_kv"]), eps=w.rms_eps)
    torch.cuda.synchronize()
    assert cache.frames_written == oc.frames_written
    return cache, oc


def window_forward(w, cache, q_c, q_r, q_pos):
    nq = q_c.shape[1]
    ws = torch.empty(V.mla_window_workspace_bytes(cache.cfg, nq), dtype=torch.uint8,
                     device="cuda")
    o = torch.empty(w.batch, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_window_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(),
                                   synth.frame_coords(w).cuda(), ws, o)
    torch.cuda.synchronize()
    return o


def oracle_window(w, oc, q_c, q_r, q_pos, tokens=None):
    out = []
    for b in range(w.batch):
        qc, qr, qp = f64(q_c[b]), f64(q_r[b]), q_pos[b].numpy()
        if tokens is not None:
            qc, qr, qp = qc[tokens], qr[tokens], qp[tokens]
        out.append(O.window_attention(oc, b, qc, qr, qp, w.head_dim, spec_of(w)))
    return np.stack(out)


# ------------------------------------------------------------------ append
SINK_SCHEDULES = [
    # mixed chunk sizes, the current chunk rewritten once
    ([(0, 2), (2, 2), (4, 1), (5, 3), (8, 3), (8, 3), (11, 2)], [0, 10, 11, 12]),
    # every append as long as the rule allows: the sink and all W - S FIFO
    # frames at once, then exactly W - S FIFO frames per call
    ([(0, 4), (4, 3), (7, 3), (7, 3), (10, 3)], [0, 10, 11, 12]),
]


@pytest.mark.parametrize("sched", range(len(SINK_SCHEDULES)))
@pytest.mark.parametrize("flags,batch", [(0, 2), (V.MLA_FLAG_SIMT, 2), (0, 64), (0, 160)])
def test_sink_fifo_slots_bit_exact(flags, batch, sched):
    """One-hot projections, no RMSNorm: every stored value is an input value,
    so the sink + FIFO slot map and the unrotated k^R match bit for bit. An
    append of more than W - S frames past the sinks is refused. Batches 2, 64
    and 160 take the tensor-core append's cluster, one-CTA-per-tile and
    two-CTAs-per-SM forms (slot runs break at the sink boundary and the FIFO
    wrap inside token tiles)."""
    schedule, expect_held = SINK_SCHEDULES[sched]
    w = synth.workload("tiny", grid_h=6, grid_w=7, window_frames=4, sink_frames=1, batch=batch)
    cfg = V.make_config(w, flags | V.MLA_FLAG_NO_RMSNORM)
    assert cfg.flags & V.MLA_FLAG_ROTATE_AT_USE
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    d, dc, dr = w.hidden, w.d_c, w.d_r
    w_dkv = torch.zeros(dc, d, dtype=torch.bfloat16)
    w_dkv[torch.arange(dc), torch.arange(dc)] = 1
    w_kr = torch.zeros(dr, d, dtype=torch.bfloat16)
    w_kr[torch.arange(dr), dc + torch.arange(dr)] = 1
    T = w.tokens_per_frame
    frames = {}
    for i, (first, n) in enumerate(schedule):
        x = synth.draw_tokens(w, n * T, 800 + i)
        V.mla_cache_append(cache, x.cuda(), w_dkv.cuda(), None, w_kr.cuda(), None, first, n)
        for k in range(n):
            frames[first + k] = x[:, k * T:(k + 1) * T]
    torch.cuda.synchronize()
    last = cache.frames_written
    with pytest.raises(V.MlaError) as e:              # frames last-3 .. last: 4 > W - S
        V.mla_cache_append(cache, synth.draw_tokens(w, 4 * T, 899).cuda(), w_dkv.cuda(), None,
                           w_kr.cuda(), None, last - 3, 4)
    assert e.value.code == V.MLA_ERR_RANGE and cache.frames_written == last
    held = O.sink_window_frames(cache.frames_written, w.window_frames, 1)
    assert held == expect_held
    c_bits = cache.c.cpu().view(torch.int16)
    k_bits = cache.kr.cpu().view(torch.int16)
    for f in held:
        s0 = O.sink_ring_slot(f, 0, T, w.window_frames, 1)
        xb = frames[f].view(torch.int16)
        assert torch.equal(c_bits[:, s0:s0 + T], xb[:, :, :dc]), f
        assert torch.equal(k_bits[:, s0:s0 + T], xb[:, :, dc:dc + dr]), f


@pytest.mark.parametrize("flags", [0, V.MLA_FLAG_SIMT])
def test_unrotated_append_values(flags):
    w = synth.workload("tiny", grid_h=10, grid_w=10, window_frames=5, sink_frames=1, batch=2,
                       rope_pairs=(6, 5, 5))
    weights = synth.draw_layer_weights(w, seed=81)
    cache, oc = window_chunks(w, weights, [(0, 3), (3, 3), (6, 2)], flags)
    valid = oc.valid_slots()
    assert oc.held_frames() == [0, 4, 5, 6, 7]
    assert_close(f64(cache.c)[:, valid], oc.c[:, valid], what="c")
    assert_close(f64(cache.kr)[:, valid], oc.kr[:, valid], what="unrotated k^R")


# --------------------------------------------------------------- attention
@pytest.mark.parametrize("flags", [0, V.MLA_FLAG_SIMT])
@pytest.mark.parametrize("case", [
    dict(grid_h=8, grid_w=8, chunks=[(0, 1), (1, 1), (2, 1)]),                 # nothing evicted
    dict(grid_h=8, grid_w=8, chunks=[(f, 1) for f in range(9)]),              # sink + 3 newest
    dict(grid_h=10, grid_w=10, chunks=[(0, 2), (2, 2), (4, 2), (6, 2), (8, 2)]),  # T = 100
])
def test_sink_window_attention_parity(case, flags):
    case = dict(case)
    chunks = case.pop("chunks")
    w = synth.workload("tiny", window_frames=4, sink_frames=1, batch=2, **case)
    weights = synth.draw_layer_weights(w, seed=82)
    cache, oc = window_chunks(w, weights, chunks, flags)
    last_first, last_n = chunks[-1]
    nq = last_n * w.tokens_per_frame
    q_c, q_r = synth.draw_queries(w, nq, 83)
    q_pos = synth.grid_positions(w, last_first, last_n)
    o = window_forward(w, cache, q_c, q_r, q_pos)
    assert_close(f64(o), oracle_window(w, oc, q_c, q_r, q_pos), what="window o_lat")


@pytest.mark.parametrize("d_c,d_r,pairs,dims", [(128, 64, (12, 10, 10), (64, 64, 64)),
                                               (64, 32, (6, 5, 5), (44, 42, 42)),
                                               (192, 64, (12, 10, 10), (64, 64, 64)),
                                               (256, 32, (6, 5, 5), (44, 42, 42)),
                                               (256, 64, (12, 10, 10), (64, 64, 64)),
                                               (512, 32, (6, 5, 5), (44, 42, 42))])
def test_sink_window_other_latent_sizes(d_c, d_r, pairs, dims):
    """The window path at other (d_c, d_r): the assembly kernel's 16-byte
    pieces per key and the tensor-core attention instance for that shape."""
    w = synth.workload("tiny", grid_h=9, grid_w=10, window_frames=4, sink_frames=1, batch=2,
                       d_c=d_c, d_r=d_r, rope_pairs=pairs, rope_axis_dims=dims)
    weights = synth.draw_layer_weights(w, seed=87)
    chunks = [(f, 1) for f in range(8)]
    cache, oc = window_chunks(w, weights, chunks)
    T = w.tokens_per_frame
    q_c, q_r = synth.draw_queries(w, T, 88)
    q_pos = synth.grid_positions(w, 7, 1)
    o = window_forward(w, cache, q_c, q_r, q_pos)
    assert_close(f64(o), oracle_window(w, oc, q_c, q_r, q_pos), what=f"window o_lat {d_c}/{d_r}")


def test_sink_window_with_one_fifo_slot():
    """S = W - 1: two sink frames and a FIFO of one frame, rolled to frame 8."""
    w = synth.workload("tiny", window_frames=3, sink_frames=2, batch=2)
    weights = synth.draw_layer_weights(w, seed=89)
    chunks = [(f, 1) for f in range(9)]
    cache, oc = window_chunks(w, weights, chunks)
    assert oc.held_frames() == [0, 1, 8]
    T = w.tokens_per_frame
    q_c, q_r = synth.draw_queries(w, T, 90)
    q_pos = synth.grid_positions(w, 8, 1)
    o = window_forward(w, cache, q_c, q_r, q_pos)
    assert_close(f64(o), oracle_window(w, oc, q_c, q_r, q_pos), what="S = W - 1")


def test_contiguous_window_matches_rotate_at_append_path():
    """No sink: re-indexed rotate-at-use attention equals the rotate-at-append
    hot path on the same inputs (RoPE relativity), after the ring wrapped."""
    w = synth.workload("tiny", grid_h=9, grid_w=11, window_frames=4, batch=2)
    weights = synth.draw_layer_weights(w, seed=84)
    dev = {k: v.cuda() for k, v in weights.items()}
    hot = V.LatentCache(V.make_config(w))
    use = V.LatentCache(V.make_config(w, V.MLA_FLAG_ROTATE_AT_USE))
    V.mla_cache_reset(hot)
    V.mla_cache_reset(use)
    T = w.tokens_per_frame
    for first in range(0, 10, 2):
        x = synth.draw_tokens(w, 2 * T, 850 + first).cuda()
        pos = synth.grid_positions(w, first, 2).cuda()
        V.mla_cache_append(hot, x, dev["w_dkv"], dev["gamma_kv"], dev["w_kr"], pos, first, 2)
        V.mla_cache_append(use, x, dev["w_dkv"], dev["gamma_kv"], dev["w_kr"], None, first, 2)
    q_c, q_r = synth.draw_queries(w, 2 * T, 86)
    q_pos = synth.grid_positions(w, 8, 2)
    o_hot = torch.empty(w.batch, 2 * T, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(hot, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o_hot)
    o_use = window_forward(w, use, q_c, q_r, q_pos)
    assert torch.equal(hot.c, use.c)
    assert_close(f64(o_use), f64(o_hot), what="rotate-at-use vs rotate-at-append")


def test_paper_rollout_window_to_frame_960():
    """The paper's long-rollout window at the Wan-1.3B frame size: one sink
    frame plus six local frames, batch 4, frames to 960; oracle on sampled
    query tokens of the last chunk."""
    w = synth.workload("sink")
    T = w.tokens_per_frame
    weights = synth.draw_layer_weights(w, seed=87)
    dev = {k: v.cuda() for k, v in weights.items()}
    cache = V.LatentCache(V.make_config(w))
    V.mla_cache_reset(cache)
    oc = O.OracleCache(w.batch, T, w.window_frames, w.d_c, w.d_r, sink_frames=1)

    def both(first, seed):
        x = synth.draw_tokens(w, 3 * T, seed)
        V.mla_cache_append(cache, x.cuda(), dev["w_dkv"], dev["gamma_kv"], dev["w_kr"], None,
                           first, 3)
        O.cache_append(oc, f64(x), f64(weights["w_dkv"]), f64(weights["w_kr"]),
                       synth.grid_positions(w, first, 3).numpy(), first, 3,
                       gamma=f64(weights["gamma_kv"]), eps=w.rms_eps)

    both(0, 880)                                       # holds the sink frame 0
    xz = torch.randn(w.batch, 3 * T, w.hidden, device="cuda").to(torch.bfloat16)
    for first in range(3, 954, 3):                     # evicted before the check
        V.mla_cache_append(cache, xz, dev["w_dkv"], dev["gamma_kv"], dev["w_kr"], None, first, 3)
    oc.frames_written = 954
    both(954, 881)
    both(957, 882)
    assert cache.frames_written == 960 and oc.held_frames() == [0] + list(range(954, 960))
    q_c, q_r = synth.draw_queries(w, 3 * T, 89)
    q_pos = synth.grid_positions(w, 957, 3)
    o = window_forward(w, cache, q_c, q_r, q_pos)
    tokens = np.arange(0, 3 * T, 31)
    ref = oracle_window(w, oc, q_c, q_r, q_pos, tokens)
    assert_close(f64(o)[:, tokens], ref, what="sink rollout o_lat")


def test_query_frame_outside_window_sets_device_status():
    w = synth.workload("tiny", window_frames=4, sink_frames=1, batch=1)
    weights = synth.draw_layer_weights(w, seed=90)
    cache, _oc = window_chunks(w, weights, [(f, 1) for f in range(8)])
    q_c, q_r = synth.draw_queries(w, w.tokens_per_frame, 91)
    q_pos = synth.grid_positions(w, 3, 1)              # frame 3 was evicted
    window_forward(w, cache, q_c, q_r, q_pos)
    assert V.mla_device_status(clear=True) == V.MLA_ERR_RANGE
    assert V.mla_device_status(clear=True) == V.MLA_OK

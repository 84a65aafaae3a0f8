"""Failure handling and resume on the GPU, without faulting it:
- a bounded device wait runs out (nothing arrives on its barrier): the
  kernel records MLA_ERR_TIMEOUT and returns, and the context keeps working;
- the cache is the only state the path carries: copying it out and back in
  (a checkpoint) and continuing reproduces the uninterrupted rollout bit for
  bit."""

import numpy as np
import pytest
import torch

from oracle import mla_oracle as O
from paper_2605_30351_gb300 import synth
from paper_2605_30351_gb300 import videomla as V

from test_gpu_parity import assert_close, f64, spec_of, upload_cache

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    V.load()
    V.mla_device_status(clear=True)
    yield
    assert V.mla_device_status(clear=True) == V.MLA_OK


def test_bounded_wait_times_out_and_context_survives():
    V.mla_device_status(clear=True)
    V.mla_selftest_bounded_wait(20_000_000)  # 20 ms
    torch.cuda.synchronize()
    assert V.mla_device_status(clear=True) == V.MLA_ERR_TIMEOUT
    # the context is still usable: an attention call afterwards is correct
    w = synth.workload("tiny", batch=1)
    cache, c, k = upload_cache(w, 97, w.window_frames)
    q_c, q_r = synth.draw_queries(w, 64, 98)
    q_pos = synth.grid_positions(w, w.window_frames - 1, 1)
    o = torch.empty(1, 64, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    ref = O.latent_attention(f64(q_c[0]), f64(q_r[0]), q_pos[0].numpy(), c[0, :cache.n_valid()],
                             k[0, :cache.n_valid()], w.head_dim, spec_of(w))
    assert_close(f64(o[0]), ref, what="attention after a timed-out wait")
    assert V.mla_device_status(clear=True) == V.MLA_OK


@pytest.mark.parametrize("sink", [0, 1])
def test_checkpoint_and_resume_reproduce_the_rollout(sink):
    w = synth.workload("tiny", grid_h=6, grid_w=9, window_frames=4, sink_frames=sink, batch=2)
    weights = {n: t.cuda() for n, t in synth.draw_layer_weights(w, 99).items()}
    T = w.tokens_per_frame
    chunks = [(f, 1) for f in range(10)]
    xs = [synth.draw_tokens(w, T, 500 + i).cuda() for i in range(len(chunks))]
    q_c, q_r = synth.draw_queries(w, T, 77)
    q_c, q_r = q_c.cuda(), q_r.cuda()

    def append(cache, i):
        first, n = chunks[i]
        pos = None if sink else synth.grid_positions(w, first, n).cuda()
        V.mla_cache_append(cache, xs[i], weights["w_dkv"], weights["gamma_kv"], weights["w_kr"],
                           pos, first, n)

    def attend(cache):
        o = torch.empty(w.batch, T, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
        q_pos = synth.grid_positions(w, cache.frames_written - 1, 1).cuda()
        if sink:
            ws = torch.empty(V.mla_window_workspace_bytes(cache.cfg, T), dtype=torch.uint8,
                             device="cuda")
            V.mla_attention_window_forward(cache, q_c, q_r, q_pos, synth.frame_coords(w).cuda(),
                                           ws, o)
        else:
            V.mla_attention_forward(cache, q_c, q_r, q_pos, o)
        return o

    cfg = V.make_config(w)
    live = V.LatentCache(cfg)
    V.mla_cache_reset(live)
    for i in range(6):
        append(live, i)
    torch.cuda.synchronize()
    ckpt = {"c": live.c.cpu(), "kr": live.kr.cpu(), "frames_written": live.frames_written}
    for i in range(6, 10):
        append(live, i)
    o_live = attend(live)
    # resume from the checkpoint in a fresh cache
    resumed = V.LatentCache(V.make_config(w))
    resumed.c.copy_(ckpt["c"])
    resumed.kr.copy_(ckpt["kr"])
    resumed.frames_written = ckpt["frames_written"]
    for i in range(6, 10):
        append(resumed, i)
    o_res = attend(resumed)
    torch.cuda.synchronize()
    assert torch.equal(live.c, resumed.c) and torch.equal(live.kr, resumed.kr)
    assert torch.equal(o_live, o_res)

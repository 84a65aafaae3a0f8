"""Large batches at the Wan-1.3B shape (64 independent sequences): the
per-batch offsets of the append and of the attention (grid rows, 64-bit
addressing past 4 GB of queries) against the float64 oracle on sampled
tokens and rows of a few batch elements."""

import numpy as np
import pytest
import torch

from oracle import mla_oracle as O
from paper_2605_30351_gb300 import synth
from paper_2605_30351_gb300 import videomla as V

from test_gpu_parity import assert_close, f64, spec_of

pytestmark = pytest.mark.gpu
B = 64
CHECK = (0, 37, B - 1)


@pytest.fixture(scope="module")
def setup():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    V.load()
    V.mla_device_status(clear=True)
    w = synth.workload("wan", batch=B)
    wt = synth.draw_layer_weights(w, seed=201)
    cache = V.LatentCache(V.make_config(w))
    V.mla_cache_reset(cache)
    g = torch.Generator(device="cuda").manual_seed(202)
    # frames 0 .. 17 as seeded device rows, then the newest chunk through the append
    cache.c.normal_(generator=g)
    cache.kr.normal_(generator=g)
    cache.frames_written = 18
    x = torch.randn(B, w.chunk_tokens, w.hidden, device="cuda", generator=g).to(torch.bfloat16)
    pos = synth.grid_positions(w, 18, 3).cuda()
    dev = {k: v.cuda() for k, v in wt.items()}
    V.mla_cache_append(cache, x, dev["w_dkv"], dev["gamma_kv"], dev["w_kr"], pos, 18, 3)
    torch.cuda.synchronize()
    yield w, wt, cache, x, pos
    assert V.mla_device_status(clear=True) == V.MLA_OK


def test_append_at_batch_64(setup):
    w, wt, cache, x, pos = setup
    tok = np.array([0, 1, 1559, 1560, 3333, w.chunk_tokens - 1])
    for b in CHECK:
        xb = f64(x[b, tok])
        c_ref = O.rmsnorm(xb @ f64(wt["w_dkv"]).T, f64(wt["gamma_kv"]), w.rms_eps)
        k_ref = O.rope3d(xb @ f64(wt["w_kr"]).T, pos[b, tok].cpu().numpy(), spec_of(w))
        slots = [O.ring_slot(18 + t // w.tokens_per_frame, t % w.tokens_per_frame,
                             w.tokens_per_frame, w.window_frames) for t in tok]
        assert_close(f64(cache.c[b, slots]), c_ref, what=f"c, batch {b}")
        assert_close(f64(cache.kr[b, slots]), k_ref, what=f"k, batch {b}")


def test_attention_at_batch_64(setup):
    w, _wt, cache, _x, pos = setup
    g = torch.Generator(device="cuda").manual_seed(203)
    q_c = (torch.randn(B, w.chunk_tokens, w.heads, w.d_c, device="cuda", generator=g)
           * (96 / 192) ** 0.5).to(torch.bfloat16)
    q_r = torch.randn(B, w.chunk_tokens, w.heads, w.d_r, device="cuda", generator=g).to(
        torch.bfloat16)
    o = torch.empty_like(q_c)
    V.mla_attention_forward(cache, q_c, q_r, pos, o)
    torch.cuda.synchronize()
    tok = np.array([0, 2500, w.chunk_tokens - 1])
    for b in CHECK:
        ref = O.latent_attention(f64(q_c[b, tok]), f64(q_r[b, tok]), pos[b, tok].cpu().numpy(),
                                 f64(cache.c[b]), f64(cache.kr[b]), w.head_dim, spec_of(w))
        assert_close(f64(o[b, tok]), ref, what=f"o_lat, batch {b}")

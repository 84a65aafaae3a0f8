"""Large batches at the Wan-1.3B shape, up to the memory-cap sweep's maxima
(the batch-scaling experiment under a fixed memory budget, Sec. 4): 64
sequences at d_c = 192, and the sweep's largest batches under its 180 GB
budget, 348 sequences at d_c = 192 and 763 at d_c = 64 (bench.memcap_plan).
At 763 the queries and the latent output are 5.5 GB each and the activations
11 GB, so the append's and the attention's per-batch offsets run past 4 GB.
For the first, a middle and the last batch element:
  attention  sampled (token, head) rows against the float64 oracle over the
             seeded cache rows (drawn on the device by a seeded generator,
             written by no kernel of the library), checked row by row
  append     the cache rows the append then writes for the newest chunk
             against RMSNorm(W_dkv x) and RoPE3D(W_kr x) of the seeded
             activations (Eq. ckv, Eq. krope, App. D.2)."""

import numpy as np
import pytest
import torch

import bench
from oracle import mla_oracle as O
from paper_2605_30351_gb300 import synth
from paper_2605_30351_gb300 import videomla as V

from test_gpu_parity import assert_close, assert_rows_close, f64, spec_of

pytestmark = pytest.mark.gpu
BUDGET = 180e9  # the memory-cap sweep's default budget (bench.py --sweep memcap)


def memcap_batch(d_c):
    w = synth.workload("wan", d_c=d_c)
    return bench.memcap_plan(w, "mla", BUDGET)["max_batch"]


CASES = [(64, 192), (memcap_batch(192), 192), (memcap_batch(64), 64)]


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    V.load()
    V.mla_device_status(clear=True)
    yield
    assert V.mla_device_status(clear=True) == V.MLA_OK


def test_memcap_batches_are_the_sweeps():
    assert CASES[1] == (348, 192) and CASES[2] == (763, 64)


@pytest.mark.parametrize("B,d_c", CASES, ids=[f"B{b}-dc{d}" for b, d in CASES])
def test_attention_then_append_at_large_batch(B, d_c):
    w = synth.workload("wan", batch=B, d_c=d_c)
    seed = 200 + B + d_c
    check = (0, B // 2, B - 1)
    nq = w.chunk_tokens
    cache = V.LatentCache(V.make_config(w))
    synth.fill_normal_(cache.c, seed)
    synth.fill_normal_(cache.kr, seed + 1)
    cache.frames_written = w.window_frames
    q_c = synth.fill_normal_(torch.empty(B, nq, w.heads, d_c, dtype=torch.bfloat16,
                                         device="cuda"), seed + 2, ((w.head_dim - w.d_r) / d_c) ** 0.5)
    q_r = synth.fill_normal_(torch.empty(B, nq, w.heads, w.d_r, dtype=torch.bfloat16,
                                         device="cuda"), seed + 3)
    pos = synth.grid_positions(w, 18, 3).cuda()
    o = torch.empty_like(q_c)
    if B == CASES[2][0]:
        assert q_c.numel() * 2 > 4 * 2 ** 30 and o.numel() * 2 > 4 * 2 ** 30
    V.mla_attention_forward(cache, q_c, q_r, pos, o)
    torch.cuda.synchronize()
    tok = np.array([0, 10, 2340, nq - 1])
    for b in check:
        ref = O.latent_attention(f64(q_c[b, tok]), f64(q_r[b, tok]), pos[b, tok].cpu().numpy(),
                                 f64(cache.c[b]), f64(cache.kr[b]), w.head_dim, spec_of(w))
        assert_rows_close(f64(o[b, tok]), ref, f"o_lat, batch {b} of {B}")
    del q_c, q_r, o

    # the append of the newest chunk (frames 18..20) into the same cache
    wt = synth.draw_layer_weights(w, seed=seed + 4)
    dev = {k: v.cuda() for k, v in wt.items()}
    x = synth.fill_normal_(torch.empty(B, nq, w.hidden, dtype=torch.bfloat16, device="cuda"),
                           seed + 5)
    V.mla_cache_append(cache, x, dev["w_dkv"], dev["gamma_kv"], dev["w_kr"], pos, 18, 3)
    torch.cuda.synchronize()
    tok = np.array([0, 1, 1559, 1560, 3333, nq - 1])
    for b in check:
        xb = f64(x[b, tok])
        c_ref = O.rmsnorm(xb @ f64(wt["w_dkv"]).T, f64(wt["gamma_kv"]), w.rms_eps)
        k_ref = O.rope3d(xb @ f64(wt["w_kr"]).T, pos[b, tok].cpu().numpy(), spec_of(w))
        slots = [O.ring_slot(18 + t // w.tokens_per_frame, t % w.tokens_per_frame,
                             w.tokens_per_frame, w.window_frames) for t in tok]
        assert_close(f64(cache.c[b, slots]), c_ref, what=f"c, batch {b} of {B}")
        assert_close(f64(cache.kr[b, slots]), k_ref, what=f"k, batch {b} of {B}")
    del x, cache
    torch.cuda.empty_cache()

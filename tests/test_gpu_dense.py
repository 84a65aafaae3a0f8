"""GPU parity of the dense per-head baseline (the cache layout VideoMLA
replaces) against the float64 oracle's textbook attention."""

import numpy as np
import pytest
import torch

from oracle import mla_oracle as O
from paper_2605_30351_gb300 import synth
from paper_2605_30351_gb300 import videomla as V

from test_gpu_parity import assert_close, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    V.load()
    V.mla_device_status(clear=True)
    yield
    assert V.mla_device_status(clear=True) == V.MLA_OK


def draw_dense(w, nq, slots, seed):
    rng = np.random.default_rng(seed)
    H, dh = w.heads, w.head_dim
    q = synth.bf16(rng.standard_normal((w.batch, nq, H, dh)))
    k = synth.bf16(rng.standard_normal((w.batch, H, slots, dh)))
    v = synth.bf16(rng.standard_normal((w.batch, H, slots, dh)))
    return q, k, v


@pytest.mark.parametrize("nq,slots,n_valid,batch,head_dim", [
    (64, 256, 256, 1, 128),     # the tiny config's shape
    (300, 500, 387, 2, 128),    # ragged tiles and a partially valid window
    (300, 500, 387, 2, 64),     # the d_h = 64 instance
])
def test_dense_attention_matches_oracle(nq, slots, n_valid, batch, head_dim):
    w = synth.workload("tiny", batch=batch, head_dim=head_dim)
    q, k, v = draw_dense(w, nq, slots, 17)
    o = torch.empty_like(q, device="cuda")
    V.mla_dense_attention_forward(V.make_config(w), q.cuda(), k.cuda(), v.cuda(), n_valid, o)
    torch.cuda.synchronize()
    ref = np.stack([O.dense_attention(f64(q[b]), f64(k[b, :, :n_valid]), f64(v[b, :, :n_valid]),
                                      w.head_dim) for b in range(batch)])
    assert_close(f64(o), ref, what="dense o")


def test_dense_attention_wan_shape_sampled_rows():
    w = synth.workload("wan")
    q, k, v = draw_dense(w, w.chunk_tokens, w.slots, 19)
    o = torch.empty_like(q, device="cuda")
    V.mla_dense_attention_forward(V.make_config(w), q.cuda(), k.cuda(), v.cuda(), w.slots, o)
    torch.cuda.synchronize()
    rows = np.array([0, 1, 777, 2500, 4001, w.chunk_tokens - 1])
    ref = O.dense_attention(f64(q[0, rows]), f64(k[0]), f64(v[0]), w.head_dim)
    assert_close(f64(o[0, rows]), ref, what="dense o at the Wan shape")


# ------------------------------------------------- decompress-then-dense
def _upload_cache(w, seed):
    cache = V.LatentCache(V.make_config(w))
    c, k = synth.draw_cache_rows(w, w.slots, seed)
    cache.c.copy_(c)
    cache.kr.copy_(k)
    cache.frames_written = w.window_frames
    return cache, f64(c), f64(k)


def _decompress(w, cache, wt):
    shape = (w.batch, w.heads, w.slots, w.head_dim)
    k = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
    v = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
    V.mla_decompress_window(cache, wt["w_uk"].cuda(), wt["w_uv"].cuda(), k, v)
    torch.cuda.synchronize()
    return k, v


@pytest.mark.parametrize("name,kw,slots_checked", [
    ("tiny", dict(grid_h=10, grid_w=10, window_frames=5, batch=2), None),   # 500 slots: ragged
    ("wan", dict(), [0, 1, 127, 128, 16001, 32759]),                        # Wan window, sampled
])
def test_decompress_reconstructs_per_head_keys_and_values(name, kw, slots_checked):
    """Eq. (reconstruct): k_h = [W_up,h^K c | k], v_h = W_up,h^V c for every slot."""
    w = synth.workload(name, **kw)
    wt = synth.draw_layer_weights(w, seed=61)
    cache, c, kr = _upload_cache(w, 62)
    k, v = _decompress(w, cache, wt)
    sl = np.arange(w.slots) if slots_checked is None else np.array(slots_checked)
    dn = w.head_dim - w.d_r
    k_nope = np.einsum("hec,bjc->bhje", f64(wt["w_uk"]), c[:, sl])
    v_ref = np.einsum("hvc,bjc->bhjv", f64(wt["w_uv"]), c[:, sl])
    kg, vg = k[:, :, sl].cpu(), v[:, :, sl].cpu()
    assert_close(f64(kg[..., :dn]), k_nope, what="k_nope")
    assert_close(f64(vg), v_ref, what="v")
    # the positional part is the cached key itself, copied for every head
    rope_bits = kg[..., dn:].view(torch.int16)
    src = cache.kr.cpu()[:, sl].view(torch.int16)
    for h in range(w.heads):
        assert torch.equal(rope_bits[:, h], src)


@pytest.mark.parametrize("d_c,d_r,pairs", [(64, 32, (6, 5, 5)), (128, 32, (6, 5, 5)),
                                        (256, 32, (6, 5, 5)), (128, 64, (12, 10, 10)),
                                        (256, 64, (12, 10, 10))])
def test_decompress_other_latent_sizes(d_c, d_r, pairs):
    """The decompression's other instances on a ragged 500-slot window, batch 2."""
    w = synth.workload("tiny", grid_h=10, grid_w=10, window_frames=5, batch=2, d_c=d_c, d_r=d_r,
                       rope_pairs=pairs)
    wt = synth.draw_layer_weights(w, seed=63 + d_c + d_r)
    cache, c, kr = _upload_cache(w, 64 + d_c)
    k, v = _decompress(w, cache, wt)
    dn = w.head_dim - w.d_r
    k_nope = np.einsum("hec,bjc->bhje", f64(wt["w_uk"]), c)
    v_ref = np.einsum("hvc,bjc->bhjv", f64(wt["w_uv"]), c)
    assert_close(f64(k[..., :dn]), k_nope, what=f"k_nope d_c={d_c} d_r={d_r}")
    assert_close(f64(v), v_ref, what=f"v d_c={d_c} d_r={d_r}")
    rope_bits = k[..., dn:].cpu().view(torch.int16)
    src = cache.kr.cpu().view(torch.int16)
    for h in range(w.heads):
        assert torch.equal(rope_bits[:, h], src)


def test_decompress_then_dense_matches_non_absorbed_oracle():
    """x -> GPU append -> decompress -> dense attention with per-head queries
    [q^nope | RoPE(q^R)], against the oracle's non-absorbed forward (Sec. 3.3)."""
    from test_gpu_parity import spec_of

    w = synth.workload("tiny", grid_h=8, grid_w=10, window_frames=3, chunk_frames=1, batch=2)
    wt = synth.draw_layer_weights(w, seed=63)
    dev = {k: v.cuda() for k, v in wt.items()}
    cache = V.LatentCache(V.make_config(w))
    V.mla_cache_reset(cache)
    T = w.tokens_per_frame
    xs, ps = [], []
    for f in range(4):                                   # frame 0 is evicted
        x = synth.draw_tokens(w, T, 64 + f)
        pos = synth.grid_positions(w, f, 1)
        V.mla_cache_append(cache, x.cuda(), dev["w_dkv"], dev["gamma_kv"], dev["w_kr"],
                           pos.cuda(), f, 1)
        xs.append(x)
        ps.append(pos)
    k, v = _decompress(w, cache, wt)
    w64 = {name: f64(t) for name, t in wt.items()}
    spec = spec_of(w)
    x_q, pos_q = xs[-1], ps[-1]
    q = []
    for b in range(w.batch):
        c_q = O.rmsnorm(f64(x_q[b]) @ w64["w_dq"].T, w64["gamma_q"], w.rms_eps)
        q_nope = np.einsum("heq,nq->nhe", w64["w_uq"], c_q)
        q_rope = O.rope3d(np.einsum("hrq,nq->nhr", w64["w_qr"], c_q), pos_q[b].numpy()[:, None],
                          spec)
        q.append(np.concatenate([q_nope, q_rope], axis=-1))
    q = synth.bf16(np.stack(q)).cuda()
    o = torch.empty_like(q)
    V.mla_dense_attention_forward(cache.cfg, q, k, v, cache.n_valid(), o)
    torch.cuda.synchronize()
    refs = []
    for b in range(w.batch):
        x_kv = np.concatenate([f64(xs[f][b]) for f in (1, 2, 3)])
        pos_kv = np.concatenate([ps[f][b].numpy() for f in (1, 2, 3)])
        refs.append(O.reference_attention(f64(x_q[b]), pos_q[b].numpy(), x_kv, pos_kv,
                                          {n: t for n, t in w64.items() if n != "w_o"},
                                          w.head_dim, spec, eps=w.rms_eps))
    assert_close(f64(o), np.stack(refs), what="decompress-then-dense o")


def test_decompress_refuses_rotate_at_use_cache():
    w = synth.workload("tiny", window_frames=4, sink_frames=1)
    cache = V.LatentCache(V.make_config(w))
    wt = synth.draw_layer_weights(w, seed=65)
    shape = (w.batch, w.heads, w.slots, w.head_dim)
    k = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(V.MlaError) as e:
        V.mla_decompress_window(cache, wt["w_uk"].cuda(), wt["w_uv"].cuda(), k, torch.empty_like(k))
    assert e.value.code == V.MLA_ERR_ARG

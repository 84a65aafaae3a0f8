"""GPU parity of the full attention layer around the latent attention:
load-time absorption (App. E), the query prologue (Eqs. cq, qnope, qrope with
RMSNorm, App. D.2) and the output projection (Eq. absorb-v), ending with the
layer output y compared against the oracle's non-absorbed training-time
forward (Sec. 3.3)."""

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


def weights64(wt):
    return {k: f64(v) for k, v in wt.items()}


def test_absorbed_weights_match_oracle():
    w = synth.workload("tiny")
    wt = synth.draw_layer_weights(w, seed=71)
    dev = {k: v.cuda() for k, v in wt.items()}
    cfg = V.make_config(w)
    w_qcat, w_b = V.mla_absorb_weights(cfg, dev["w_uq"], dev["w_uk"], dev["w_qr"],
                                       dev["gamma_q"], dev["w_uv"], dev["w_o"])
    torch.cuda.synchronize()
    w64 = weights64(wt)
    A = O.absorbed_query_matrices(w64["w_uq"], w64["w_uk"])            # [H, d_q, d_c]
    ref_qc = np.concatenate([A[h].T for h in range(w.heads)]) * w64["gamma_q"][None, :]
    ref_qr = w64["w_qr"].reshape(-1, w.d_q) * w64["gamma_q"][None, :]
    got = f64(w_qcat)
    assert_close(got[:w.heads * w.d_c], ref_qc, what="W_qc")
    assert_close(got[w.heads * w.d_c:], ref_qr, what="W_qr")
    B = O.absorbed_output_matrices(w64["w_uv"], w64["w_o"])            # [H, d, d_c]
    ref_b = np.concatenate([B[h] for h in range(w.heads)], axis=1)
    assert_close(f64(w_b), ref_b, what="W_B")


@pytest.mark.parametrize("nq,batch,shape", [
    (64, 1, {}), (200, 2, {}),
    (130, 2, dict(d_c=128, d_r=64, rope_pairs=(12, 10, 10), rope_axis_dims=(64, 64, 64))),
])
def test_query_prologue_matches_oracle(nq, batch, shape):
    w = synth.workload("tiny", batch=batch, **shape)
    wt = synth.draw_layer_weights(w, seed=72)
    dev = {k: v.cuda() for k, v in wt.items()}
    cfg = V.make_config(w)
    w_qcat, _ = V.mla_absorb_weights(cfg, dev["w_uq"], dev["w_uk"], dev["w_qr"], dev["gamma_q"],
                                     dev["w_uv"], dev["w_o"])
    x = synth.draw_tokens(w, nq, 73)
    ws = torch.empty(V.mla_query_workspace_bytes(cfg, nq), dtype=torch.uint8, device="cuda")
    q_c = torch.empty(batch, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    q_r = torch.empty(batch, nq, w.heads, w.d_r, dtype=torch.bfloat16, device="cuda")
    V.mla_query_prologue(cfg, x.cuda(), dev["w_dq"], w_qcat, ws, q_c, q_r)
    torch.cuda.synchronize()
    w64 = weights64(wt)
    c_q = O.rmsnorm(f64(x) @ w64["w_dq"].T, w64["gamma_q"], w.rms_eps)
    ref_qc = np.stack([O.absorb_query(c_q[b], w64["w_uq"], w64["w_uk"]) for b in range(batch)])
    ref_qr = np.einsum("hrq,bnq->bnhr", w64["w_qr"], c_q)
    assert_close(f64(q_c), ref_qc, what="q_c")
    assert_close(f64(q_r), ref_qr, what="q_r")


@pytest.mark.parametrize("heads,d_c", [(12, 192), (3, 64)])
def test_layer_gemms_at_four_chunks_match_oracle(heads, d_c):
    """Four Wan-1.3B chunks (18,720 query tokens): both query-prologue GEMMs and
    the output projection run the persistent paired-SM kernel (two M tiles per
    M = 256 MMA, each CTA holding half of the B rows, clusters walking the
    pair tiles; 147 M tiles, so the last pair has a tile past the tokens).
    With 3 heads of d_c = 64 the absorbed query GEMM has N = 288: its first
    256-wide tile straddles the q_c | q_r split at column 192 and its second
    is ragged, and the output projection's K (192) is three K blocks, fewer
    than the ring's stages. Sampled rows, including the first and last pair,
    against the oracle (Eqs. cq, qnope, qrope, absorb-v)."""
    w = synth.workload("wan", batch=4, heads=heads, d_c=d_c)
    nq = w.chunk_tokens
    wt = synth.draw_layer_weights(w, seed=74)
    dev = {k: v.cuda() for k, v in wt.items()}
    cfg = V.make_config(w)
    w_qcat, w_b = V.mla_absorb_weights(cfg, dev["w_uq"], dev["w_uk"], dev["w_qr"], dev["gamma_q"],
                                       dev["w_uv"], dev["w_o"])
    x = synth.draw_tokens(w, nq, 75)
    ws = torch.empty(V.mla_query_workspace_bytes(cfg, nq), dtype=torch.uint8, device="cuda")
    q_c = torch.empty(4, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    q_r = torch.empty(4, nq, w.heads, w.d_r, dtype=torch.bfloat16, device="cuda")
    V.mla_query_prologue(cfg, x.cuda(), dev["w_dq"], w_qcat, ws, q_c, q_r)
    o = synth.draw_queries(w, nq, 76)[0]          # any bf16 latent output [4, nq, H, d_c]
    y = torch.empty(4, nq, w.hidden, dtype=torch.bfloat16, device="cuda")
    V.mla_output_projection(cfg, o.cuda(), w_b, y)
    torch.cuda.synchronize()
    w64 = weights64(wt)
    B = O.absorbed_output_matrices(w64["w_uv"], w64["w_o"])            # [H, d, d_c]
    for b, toks in ((0, [0, 1, 127, 128, 255, 256, 2000]), (3, [4000, 4607, 4608, 4679])):
        xs = f64(x[b])[toks]
        c_q = O.rmsnorm(xs @ w64["w_dq"].T, w64["gamma_q"], w.rms_eps)
        assert_close(f64(q_c[b])[toks], O.absorb_query(c_q, w64["w_uq"], w64["w_uk"]),
                     what=f"q_c, chunk {b}")
        assert_close(f64(q_r[b])[toks], np.einsum("hrq,nq->nhr", w64["w_qr"], c_q),
                     what=f"q_r, chunk {b}")
        ref_y = np.einsum("hdc,nhc->nd", B, f64(o[b])[toks])
        assert_close(f64(y[b])[toks], ref_y, what=f"y, chunk {b}")


def test_full_layer_output_matches_non_absorbed_oracle():
    """x -> cache append (every window frame) -> query prologue -> latent
    attention -> output projection on the GPU, against the oracle's
    non-absorbed forward with per-head keys and values reconstructed from the
    same cache definition and W_O applied to the concatenated heads."""
    w = synth.workload("tiny", grid_h=8, grid_w=10, window_frames=3, chunk_frames=1, batch=2)
    wt = synth.draw_layer_weights(w, seed=81)
    dev = {k: v.cuda() for k, v in wt.items()}
    cfg = V.make_config(w)
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    T = w.tokens_per_frame
    xs, ps = [], []
    for f in range(4):                                   # frame 0 is evicted at the end
        x = synth.draw_tokens(w, T, 90 + f)
        pos = synth.grid_positions(w, f, 1)
        V.mla_cache_append(cache, x.cuda(), dev["w_dkv"], dev["gamma_kv"], dev["w_kr"],
                           pos.cuda(), f, 1)
        xs.append(x)
        ps.append(pos)
    w_qcat, w_b = V.mla_absorb_weights(cfg, dev["w_uq"], dev["w_uk"], dev["w_qr"],
                                       dev["gamma_q"], dev["w_uv"], dev["w_o"])
    x_q, pos_q = xs[-1], ps[-1]                          # the current chunk queries itself
    ws = torch.empty(V.mla_query_workspace_bytes(cfg, T), dtype=torch.uint8, device="cuda")
    q_c = torch.empty(w.batch, T, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    q_r = torch.empty(w.batch, T, w.heads, w.d_r, dtype=torch.bfloat16, device="cuda")
    V.mla_query_prologue(cfg, x_q.cuda(), dev["w_dq"], w_qcat, ws, q_c, q_r)
    o_lat = torch.empty_like(q_c)
    V.mla_attention_forward(cache, q_c, q_r, pos_q.cuda(), o_lat)
    y = torch.empty(w.batch, T, w.hidden, dtype=torch.bfloat16, device="cuda")
    V.mla_output_projection(cfg, o_lat, w_b, y)
    torch.cuda.synchronize()
    w64 = weights64(wt)
    refs = []
    for b in range(w.batch):
        x_kv = np.concatenate([f64(xs[f][b]) for f in (1, 2, 3)])
        pos_kv = np.concatenate([ps[f][b].numpy() for f in (1, 2, 3)])
        _o, y_ref = O.reference_attention(f64(x_q[b]), pos_q[b].numpy(), x_kv, pos_kv, w64,
                                          w.head_dim, spec_of(w), eps=w.rms_eps)
        refs.append(y_ref)
    assert_close(f64(y), np.stack(refs), what="layer output y")


@pytest.mark.parametrize("batch", [1, 4])
def test_output_projection_at_wan_size(batch):
    """y = o_lat W_B^T at one and four Wan chunks (the two tile widths the
    launcher picks between), checked on sampled rows in float64."""
    w = synth.workload("wan", batch=batch)
    wt = synth.draw_layer_weights(w, seed=95)
    dev = {k: v.cuda() for k, v in wt.items()}
    cfg = V.make_config(w)
    _w_qcat, w_b = V.mla_absorb_weights(cfg, dev["w_uq"], dev["w_uk"], dev["w_qr"], dev["gamma_q"],
                                        dev["w_uv"], dev["w_o"])
    g = torch.Generator(device="cuda").manual_seed(96)
    o_lat = torch.randn(batch, w.chunk_tokens, w.heads, w.d_c, device="cuda", generator=g)
    o_lat = o_lat.to(torch.bfloat16)
    y = torch.empty(batch, w.chunk_tokens, w.hidden, dtype=torch.bfloat16, device="cuda")
    V.mla_output_projection(cfg, o_lat, w_b, y)
    torch.cuda.synchronize()
    rows = np.array([0, 1, 127, 128, 2999, w.chunk_tokens - 1])
    flat = f64(o_lat).reshape(batch, w.chunk_tokens, -1)[:, rows]
    ref = flat @ f64(w_b).T
    assert_close(f64(y)[:, rows], ref, what=f"y, batch {batch}")


@pytest.mark.parametrize("batch", [1, 2])
def test_query_prologue_at_wan_size(batch):
    """The prologue at one and two Wan chunks (the first GEMM's two tile
    widths), checked against the oracle on sampled tokens."""
    w = synth.workload("wan", batch=batch)
    wt = synth.draw_layer_weights(w, seed=97)
    dev = {k: v.cuda() for k, v in wt.items()}
    cfg = V.make_config(w)
    w_qcat, _ = V.mla_absorb_weights(cfg, dev["w_uq"], dev["w_uk"], dev["w_qr"], dev["gamma_q"],
                                     dev["w_uv"], dev["w_o"])
    nq = w.chunk_tokens
    x = synth.draw_tokens(w, nq, 98)
    ws = torch.empty(V.mla_query_workspace_bytes(cfg, nq), dtype=torch.uint8, device="cuda")
    q_c = torch.empty(batch, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    q_r = torch.empty(batch, nq, w.heads, w.d_r, dtype=torch.bfloat16, device="cuda")
    V.mla_query_prologue(cfg, x.cuda(), dev["w_dq"], w_qcat, ws, q_c, q_r)
    torch.cuda.synchronize()
    tok = np.array([0, 1, 127, 128, 3000, nq - 1])
    w64 = weights64(wt)
    c_q = O.rmsnorm(f64(x[:, tok]) @ w64["w_dq"].T, w64["gamma_q"], w.rms_eps)
    ref_qc = np.stack([O.absorb_query(c_q[b], w64["w_uq"], w64["w_uk"]) for b in range(batch)])
    ref_qr = np.einsum("hrq,bnq->bnhr", w64["w_qr"], c_q)
    assert_close(f64(q_c[:, tok]), ref_qc, what="q_c at Wan size")
    assert_close(f64(q_r[:, tok]), ref_qr, what="q_r at Wan size")

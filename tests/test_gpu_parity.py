"""GPU parity: the CUDA path (through the C ABI) against the float64 oracle on
the same seeded inputs. Tolerance from the specification of this path:
max-abs <= 2e-2 and relative L2 <= 1e-2 for floating point; ring-buffer
indexing bit-exact."""

import numpy as np
import pytest
import torch

from oracle import mla_oracle as O
from paper_2605_30351_gb300 import synth
from paper_2605_30351_gb300 import videomla as V

pytestmark = pytest.mark.gpu

MAX_ABS = 2e-2
REL_L2 = 1e-2


def assert_close(got, ref, max_abs=MAX_ABS, rel_l2=REL_L2, what=""):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    d = got - ref
    ma = float(np.max(np.abs(d))) if d.size else 0.0
    rl = float(np.linalg.norm(d) / max(np.linalg.norm(ref), 1e-30))
    assert ma <= max_abs and rl <= rel_l2, f"{what}: max_abs={ma:.3e} rel_l2={rl:.3e}"
    return ma, rl


def assert_rows_close(got, ref, what, row_rel=1e-2):
    """Per row (last axis = one output row): rel-L2 <= row_rel and max-abs <=
    row_rel * max|ref row|; over all rows the bounds of assert_close."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    got = got.reshape(-1, got.shape[-1])
    ref = ref.reshape(-1, ref.shape[-1])
    assert_close(got, ref, what=what)
    d = got - ref
    rel = np.linalg.norm(d, axis=1) / np.maximum(np.linalg.norm(ref, axis=1), 1e-30)
    mab = np.max(np.abs(d), axis=1) / np.maximum(np.max(np.abs(ref), axis=1), 1e-30)
    worst = int(np.argmax(rel))
    assert rel.max() <= row_rel, f"{what}: row {worst} rel-L2 {rel[worst]:.3e}"
    worst = int(np.argmax(mab))
    assert mab.max() <= row_rel, f"{what}: row {worst} max-abs/max|ref| {mab[worst]:.3e}"


def f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def spec_of(w):
    return O.RopeSpec(w.rope_pairs, w.rope_axis_dims, w.rope_theta)


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    V.load()
    V.mla_device_status(clear=True)
    yield
    assert V.mla_device_status(clear=True) == V.MLA_OK


def run_chunks(w, weights, chunks, flags=0, seed=100):
    """Append `chunks` = [(first_frame, n_frames), ...] on the GPU and in the oracle."""
    cfg = V.make_config(w, flags)
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    oc = O.OracleCache(w.batch, w.tokens_per_frame, w.window_frames, w.d_c, w.d_r)
    dev = {k: v.cuda() for k, v in weights.items()}
    for i, (first, n) in enumerate(chunks):
        x = synth.draw_tokens(w, n * w.tokens_per_frame, seed + i)
        pos = synth.grid_positions(w, first, n)
        V.mla_cache_append(cache, x.cuda(), dev["w_dkv"], dev["gamma_kv"], dev["w_kr"],
                           pos.cuda(), first, n)
        O.cache_append(oc, f64(x), f64(weights["w_dkv"]), f64(weights["w_kr"]), pos.numpy(),
                       first, n, gamma=f64(weights["gamma_kv"]), eps=w.rms_eps,
                       use_rmsnorm=not (flags & V.MLA_FLAG_NO_RMSNORM), spec=spec_of(w))
    torch.cuda.synchronize()
    assert cache.frames_written == oc.frames_written
    return cache, oc


def small(name="tiny", **kw):
    return synth.workload(name, **kw)


# ------------------------------------------------------------------ append
@pytest.mark.parametrize("flags", [0, V.MLA_FLAG_SIMT])
def test_append_parity_tiny(flags):
    w = small()
    weights = synth.draw_layer_weights(w, seed=1)
    cache, oc = run_chunks(w, weights, [(0, 1), (1, 1), (2, 1), (3, 1)], flags)
    valid = oc.valid_slots()
    assert_close(f64(cache.c)[:, valid], oc.c[:, valid], what="c")
    assert_close(f64(cache.kr)[:, valid], oc.kr[:, valid], what="k_rope")


def test_append_parity_ragged_batch2_wrap():
    # T = 100 tokens per frame (not a multiple of 128), batch 2, ring wraps
    w = small(grid_h=10, grid_w=10, window_frames=5, batch=2, rope_pairs=(6, 5, 5))
    weights = synth.draw_layer_weights(w, seed=2)
    cache, oc = run_chunks(w, weights, [(0, 3), (3, 3), (3, 3), (6, 2)])
    valid = oc.valid_slots()
    assert len(valid) == 5 * 100
    assert_close(f64(cache.c)[:, valid], oc.c[:, valid], what="c")
    assert_close(f64(cache.kr)[:, valid], oc.kr[:, valid], what="k_rope")


@pytest.mark.parametrize("batch", [2, 64, 160])
def test_ring_bit_exact(batch):
    """One-hot projections, no RMSNorm, positions at zero: every appended
    value is an input value, so slot contents must match bit for bit. With
    42 tokens per frame a token tile holds several frames (slot runs break
    inside tiles, the ring wraps inside tiles). Batch 2 takes the append's
    cluster form, 64 one CTA per tile, 160 (more tiles than SMs) two CTAs
    per SM."""
    w = small(grid_h=6, grid_w=7, window_frames=4, batch=batch)
    cfg = V.make_config(w, V.MLA_FLAG_NO_RMSNORM)
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    d, dc, dr = w.hidden, w.d_c, w.d_r
    w_dkv = torch.zeros(dc, d, dtype=torch.bfloat16)
    w_dkv[torch.arange(dc), torch.arange(dc)] = 1
    w_kr = torch.zeros(dr, d, dtype=torch.bfloat16)
    w_kr[torch.arange(dr), dc + torch.arange(dr)] = 1
    T = w.tokens_per_frame
    frames = {}
    schedule = [(0, 2), (2, 2), (4, 1), (5, 3), (8, 3), (8, 3), (11, 2)]
    for i, (first, n) in enumerate(schedule):
        x = synth.draw_tokens(w, n * T, 500 + i)
        pos = torch.zeros(w.batch, n * T, 3, dtype=torch.int32)
        V.mla_cache_append(cache, x.cuda(), w_dkv.cuda(), None, w_kr.cuda(), pos.cuda(), first, n)
        for k in range(n):
            frames[first + k] = x[:, k * T:(k + 1) * T]
    torch.cuda.synchronize()
    c_bits = cache.c.cpu().view(torch.int16)
    k_bits = cache.kr.cpu().view(torch.int16)
    for f in O.window_frames(cache.frames_written, w.window_frames):
        s0 = O.ring_slot(f, 0, T, w.window_frames)
        xb = frames[f].view(torch.int16)
        assert torch.equal(c_bits[:, s0:s0 + T], xb[:, :, :dc]), f
        assert torch.equal(k_bits[:, s0:s0 + T], xb[:, :, dc:dc + dr]), f


# --------------------------------------------------------------- attention
def upload_cache(w, seed, frames_written, flags=0):
    """Fill a cache with seeded rows (not produced by the GPU) for attention tests."""
    cfg = V.make_config(w, flags)
    cache = V.LatentCache(cfg)
    c, k = synth.draw_cache_rows(w, w.slots, seed)
    cache.c.copy_(c)
    cache.kr.copy_(k)
    cache.frames_written = frames_written
    return cache, f64(c), f64(k)


def oracle_latent(w, q_c, q_r, q_pos, c, k, n_valid, rows=None):
    out = []
    for b in range(w.batch):
        qc, qr, qp = f64(q_c[b]), f64(q_r[b]), q_pos[b].numpy()
        if rows is not None:
            tok = rows // w.heads
            o = O.latent_attention(qc[tok], qr[tok], qp[tok], c[b, :n_valid], k[b, :n_valid],
                                   w.head_dim, spec_of(w))
            out.append(o[np.arange(len(rows)), rows % w.heads])
        else:
            out.append(O.latent_attention(qc, qr, qp, c[b, :n_valid], k[b, :n_valid],
                                          w.head_dim, spec_of(w)))
    return np.stack(out)


@pytest.mark.parametrize("flags", [0, V.MLA_FLAG_SIMT])
@pytest.mark.parametrize("case", [
    dict(grid_h=8, grid_w=8, window_frames=4, fw=4, nq=64),     # tiny: 768 rows, 256 keys
    dict(grid_h=10, grid_w=10, window_frames=5, fw=3, nq=50),   # ragged: 300 keys, 600 rows
    dict(grid_h=9, grid_w=7, window_frames=3, fw=7, nq=63),     # wrapped ring, 189 keys
])
def test_attention_parity(case, flags):
    case = dict(case)
    fw, nq = case.pop("fw"), case.pop("nq")
    w = small(batch=2, **case)
    cache, c, k = upload_cache(w, 7, fw, flags)
    q_c, q_r = synth.draw_queries(w, nq, 8)
    q_pos = synth.grid_positions(w, max(fw - 1, 0), 1)[:, :nq].contiguous()
    o = torch.empty(w.batch, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    ref = oracle_latent(w, q_c, q_r, q_pos, c, k, cache.n_valid())
    assert_close(f64(o), ref, what="o_lat")


@pytest.mark.parametrize("d_c,d_r,pairs", [
    (64, 32, (4, 6, 6)), (128, 32, (6, 5, 5)), (256, 32, (6, 5, 5)),
    (64, 64, (12, 10, 10)), (128, 64, (12, 10, 10)), (192, 64, (12, 10, 10)),
    (256, 64, (12, 10, 10)),
])
def test_attention_latent_sweep(d_c, d_r, pairs):
    w = small(d_c=d_c, d_r=d_r, rope_pairs=pairs, rope_axis_dims=(44, 42, 42) if d_r == 32
              else (64, 64, 64), grid_h=10, grid_w=13, window_frames=3, batch=1)
    cache, c, k = upload_cache(w, 11, 3)
    q_c, q_r = synth.draw_queries(w, 40, 12)
    q_pos = synth.grid_positions(w, 2, 1)[:, :40].contiguous()
    o = torch.empty(1, 40, w.heads, d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    ref = oracle_latent(w, q_c, q_r, q_pos, c, k, cache.n_valid())
    assert_close(f64(o), ref, what=f"o_lat d_c={d_c} d_r={d_r}")


def test_attention_dc512_simt():
    w = small(d_c=512, d_r=32, grid_h=6, grid_w=6, window_frames=3, batch=1)
    cache, c, k = upload_cache(w, 13, 3, V.MLA_FLAG_SIMT)
    q_c, q_r = synth.draw_queries(w, 20, 14)
    q_pos = synth.grid_positions(w, 2, 1)[:, :20].contiguous()
    o = torch.empty(1, 20, w.heads, 512, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    assert_close(f64(o), oracle_latent(w, q_c, q_r, q_pos, c, k, cache.n_valid()), what="d_c=512")


# the append's two forms at every latent size with a tensor-core instance:
# small grids take clusters of d_c/64 CTAs (2, 3 or 4; x multicast in 64- or
# 32-row parts), larger ones one CTA per token tile
APPEND_SIZES = [(64, 32, (6, 5, 5), (44, 42, 42)), (128, 32, (6, 5, 5), (44, 42, 42)),
                (256, 32, (6, 5, 5), (44, 42, 42)), (64, 64, (12, 10, 10), (64, 64, 64)),
                (128, 64, (12, 10, 10), (64, 64, 64)), (256, 64, (12, 10, 10), (64, 64, 64))]


@pytest.mark.parametrize("d_c,d_r,pairs,dims", APPEND_SIZES)
@pytest.mark.parametrize("form", ["small", "large"])
def test_append_latent_sizes(d_c, d_r, pairs, dims, form):
    """small: T = 100, batch 2, ring wrap (3 token tiles per chunk: the
    cluster form for d_c >= 128); large: the Wan grid, 3-frame chunks,
    batch 3 (111 token tiles: one CTA per tile)."""
    if form == "small":
        w = small(d_c=d_c, d_r=d_r, rope_pairs=pairs, rope_axis_dims=dims, grid_h=10, grid_w=10,
                  window_frames=5, batch=2)
        chunks = [(0, 3), (3, 3), (3, 3), (6, 2)]
    else:
        w = synth.workload("wan").with_(d_c=d_c, d_r=d_r, rope_pairs=pairs, rope_axis_dims=dims,
                                        window_frames=6, batch=3)
        chunks = [(0, 3), (3, 3), (6, 3)]
    weights = synth.draw_layer_weights(w, seed=23 + d_c + d_r)
    cache, oc = run_chunks(w, weights, chunks, seed=230)
    valid = oc.valid_slots()
    assert_close(f64(cache.c)[:, valid], oc.c[:, valid], what=f"c {d_c}/{d_r} {form}")
    assert_close(f64(cache.kr)[:, valid], oc.kr[:, valid], what=f"k_rope {d_c}/{d_r} {form}")


# d_c = 512: the attention output is split over a CTA pair (256 columns
# each) and the append runs its c and k^R halves in separate CTAs
DC512 = [(32, (6, 5, 5), (44, 42, 42)), (64, (12, 10, 10), (64, 64, 64))]


@pytest.mark.parametrize("d_r,pairs,dims", DC512)
def test_append_dc512_parity(d_r, pairs, dims):
    """T = 100 (ragged tiles), batch 2, ring wrapped, RMSNorm over 512 columns."""
    w = small(d_c=512, d_r=d_r, rope_pairs=pairs, rope_axis_dims=dims, grid_h=10, grid_w=10,
              window_frames=4, batch=2)
    weights = synth.draw_layer_weights(w, seed=17)
    cache, oc = run_chunks(w, weights, [(0, 2), (2, 2), (4, 1)])
    valid = oc.valid_slots()
    assert len(valid) == 4 * 100
    assert_close(f64(cache.c)[:, valid], oc.c[:, valid], what="c d_c=512")
    assert_close(f64(cache.kr)[:, valid], oc.kr[:, valid], what="k_rope d_c=512")


def test_append_dc512_bit_exact():
    """One-hot projections, no RMSNorm, positions zero: both halves of the
    split append copy input values, so slots match bit for bit."""
    w = small(d_c=512, d_r=32, rope_pairs=(6, 5, 5), grid_h=9, grid_w=9, window_frames=3,
              batch=2)
    cfg = V.make_config(w, V.MLA_FLAG_NO_RMSNORM)
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    d, dc, dr = w.hidden, w.d_c, w.d_r
    w_dkv = torch.zeros(dc, d, dtype=torch.bfloat16)
    w_dkv[torch.arange(dc), torch.arange(dc)] = 1
    w_kr = torch.zeros(dr, d, dtype=torch.bfloat16)
    w_kr[torch.arange(dr), dc + torch.arange(dr)] = 1
    T = w.tokens_per_frame
    frames = {}
    for i, (first, n) in enumerate([(0, 2), (2, 2), (4, 1)]):
        x = synth.draw_tokens(w, n * T, 520 + i)
        pos = torch.zeros(w.batch, n * T, 3, dtype=torch.int32)
        V.mla_cache_append(cache, x.cuda(), w_dkv.cuda(), None, w_kr.cuda(), pos.cuda(), first, n)
        for k in range(n):
            frames[first + k] = x[:, k * T:(k + 1) * T]
    torch.cuda.synchronize()
    c_bits = cache.c.cpu().view(torch.int16)
    k_bits = cache.kr.cpu().view(torch.int16)
    for f in O.window_frames(cache.frames_written, w.window_frames):
        s0 = O.ring_slot(f, 0, T, w.window_frames)
        xb = frames[f].view(torch.int16)
        assert torch.equal(c_bits[:, s0:s0 + T], xb[:, :, :dc]), f
        assert torch.equal(k_bits[:, s0:s0 + T], xb[:, :, dc:dc + dr]), f


@pytest.mark.parametrize("d_r,pairs,dims", DC512)
def test_attention_dc512_parity(d_r, pairs, dims):
    """390 keys (six 64-key blocks and a ragged one), 480 rows (a ragged
    fourth row tile), batch 2."""
    w = small(d_c=512, d_r=d_r, rope_pairs=pairs, rope_axis_dims=dims, grid_h=10, grid_w=13,
              window_frames=3, batch=2)
    cache, c, k = upload_cache(w, 15, 3)
    q_c, q_r = synth.draw_queries(w, 40, 16)
    q_pos = synth.grid_positions(w, 2, 1)[:, :40].contiguous()
    o = torch.empty(w.batch, 40, w.heads, 512, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    assert_close(f64(o), oracle_latent(w, q_c, q_r, q_pos, c, k, cache.n_valid()),
                 what=f"d_c=512 d_r={d_r}")


def test_attention_dc512_wan_sampled_rows():
    """Wan shape with d_c = 512 (4680 x 12 rows, 32760 keys), sampled rows,
    including both output halves of the first and last row tiles."""
    w = synth.workload("wan").with_(d_c=512)
    cache, c, k = upload_cache(w, 35, w.window_frames)
    q_c, q_r = synth.draw_queries(w, w.chunk_tokens, 36)
    q_pos = synth.grid_positions(w, 18, 3)
    o = torch.empty(1, w.chunk_tokens, w.heads, 512, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    rng = np.random.default_rng(1)
    rows = np.sort(rng.choice(w.chunk_tokens * w.heads, 48, replace=False))
    rows = np.concatenate([[0, 127], rows, [w.chunk_tokens * w.heads - 1]])
    ref = oracle_latent(w, q_c, q_r, q_pos, c, k, cache.n_valid(), rows=rows)
    got = f64(o).reshape(1, -1, 512)[:, rows]
    assert_close(got, ref, what="d_c=512 Wan rows")


def test_tc_matches_simt_wan_rows():
    """Tensor-core and SIMT kernels agree at the full Wan-1.3B layer shape."""
    w = synth.workload("wan")
    cache, c, k = upload_cache(w, 21, w.window_frames)
    q_c, q_r = synth.draw_queries(w, w.chunk_tokens, 22)
    q_pos = synth.grid_positions(w, 18, 3)
    args = (q_c.cuda(), q_r.cuda(), q_pos.cuda())
    o_tc = torch.empty(1, w.chunk_tokens, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, *args, o_tc)
    cache.struct.cfg.flags = V.MLA_FLAG_SIMT
    o_simt = torch.empty_like(o_tc)
    V.mla_attention_forward(cache, *args, o_simt)
    torch.cuda.synchronize()
    assert_close(f64(o_tc), f64(o_simt), what="tc vs simt")


def test_attention_wan_sampled_rows():
    """Full Wan-1.3B shape (4680 x 12 rows, 32760 keys), oracle on sampled rows."""
    w = synth.workload("wan")
    cache, c, k = upload_cache(w, 31, w.window_frames)
    q_c, q_r = synth.draw_queries(w, w.chunk_tokens, 32)
    q_pos = synth.grid_positions(w, 18, 3)
    o = torch.empty(1, w.chunk_tokens, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    rng = np.random.default_rng(0)
    rows = np.sort(rng.choice(w.chunk_tokens * w.heads, 96, replace=False))
    rows = np.concatenate([rows, [0, w.chunk_tokens * w.heads - 1]])
    ref = oracle_latent(w, q_c, q_r, q_pos, c, k, w.slots, rows=rows)
    got = f64(o).reshape(1, -1, w.d_c)[:, rows]
    assert_close(got, ref, what="wan sampled")


@pytest.mark.parametrize("d_c,d_r,pairs,dims", [
    (64, 32, (6, 5, 5), (44, 42, 42)), (128, 32, (6, 5, 5), (44, 42, 42)),
    (256, 32, (6, 5, 5), (44, 42, 42)), (64, 64, (12, 10, 10), (64, 64, 64)),
    (128, 64, (12, 10, 10), (64, 64, 64)), (192, 64, (12, 10, 10), (64, 64, 64)),
    (256, 64, (12, 10, 10), (64, 64, 64)),
])
def test_attention_latent_sizes_wan_sampled_rows(d_c, d_r, pairs, dims):
    """Every tensor-core instance at the Wan shape (32,760 keys: the stage
    ring laps many times), oracle on sampled rows of the first, a middle and
    the last row tile."""
    w = synth.workload("wan").with_(d_c=d_c, d_r=d_r, rope_pairs=pairs, rope_axis_dims=dims)
    cache, c, k = upload_cache(w, 41 + d_c + d_r, w.window_frames)
    q_c, q_r = synth.draw_queries(w, w.chunk_tokens, 42 + d_c)
    q_pos = synth.grid_positions(w, 18, 3)
    o = torch.empty(1, w.chunk_tokens, w.heads, d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    rng = np.random.default_rng(d_c + d_r)
    n = w.chunk_tokens * w.heads
    rows = np.unique(np.concatenate([[0, 127, n // 2, n - 1], rng.choice(n, 20, replace=False)]))
    ref = oracle_latent(w, q_c, q_r, q_pos, c, k, cache.n_valid(), rows=rows)
    got = f64(o).reshape(1, -1, d_c)[:, rows]
    assert_close(got, ref, what=f"Wan rows d_c={d_c} d_r={d_r}")


def test_append_then_attention_chain():
    """Each side runs its own append then attention: end-to-end latent output."""
    w = small(grid_h=10, grid_w=12, window_frames=4, chunk_frames=2, batch=2)
    weights = synth.draw_layer_weights(w, seed=41)
    cache, oc = run_chunks(w, weights, [(0, 2), (2, 2), (4, 2)])
    q_c, q_r = synth.draw_queries(w, 2 * w.tokens_per_frame, 42)
    q_pos = synth.grid_positions(w, 4, 2)
    o = torch.empty(w.batch, q_c.shape[1], w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    valid = oc.valid_slots()
    ref = np.stack([O.latent_attention(f64(q_c[b]), f64(q_r[b]), q_pos[b].numpy(),
                                       oc.c[b, valid], oc.kr[b, valid], w.head_dim, spec_of(w),
                                       key_frames=oc.frame_of_slot[valid], query_last_frame=5)
                    for b in range(w.batch)])
    assert_close(f64(o), ref, what="chain")


def test_rollout_positions_to_960():
    """Batch 4, ring wrapped many times, temporal positions near 960."""
    w = small(grid_h=12, grid_w=13, window_frames=21, chunk_frames=3, batch=4,
              rope_pairs=(6, 5, 5))
    weights = synth.draw_layer_weights(w, seed=51)
    cfg = V.make_config(w)
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    dev = {k: v.cuda() for k, v in weights.items()}
    T = w.tokens_per_frame
    # frames 0 .. 938 with cheap device-side activations (evicted before the check)
    xz = torch.randn(w.batch, 3 * T, w.hidden, device="cuda").to(torch.bfloat16)
    for first in range(0, 939, 3):
        pos = synth.grid_positions(w, first, 3).cuda()
        V.mla_cache_append(cache, xz, dev["w_dkv"], dev["gamma_kv"], dev["w_kr"], pos, first, 3)
    oc = O.OracleCache(w.batch, T, w.window_frames, w.d_c, w.d_r)
    oc.frames_written = 939
    for i, first in enumerate(range(939, 960, 3)):     # the 7 chunks that stay in the window
        x = synth.draw_tokens(w, 3 * T, 600 + i)
        pos = synth.grid_positions(w, first, 3)
        V.mla_cache_append(cache, x.cuda(), dev["w_dkv"], dev["gamma_kv"], dev["w_kr"],
                           pos.cuda(), first, 3)
        O.cache_append(oc, f64(x), f64(weights["w_dkv"]), f64(weights["w_kr"]), pos.numpy(),
                       first, 3, gamma=f64(weights["gamma_kv"]), eps=w.rms_eps, spec=spec_of(w))
    assert cache.frames_written == 960
    valid = oc.valid_slots()
    assert len(valid) == w.slots
    assert_close(f64(cache.c)[:, valid], oc.c[:, valid], what="c at t~960")
    assert_close(f64(cache.kr)[:, valid], oc.kr[:, valid], what="k_rope at t~960")
    q_c, q_r = synth.draw_queries(w, 3 * T, 61)
    q_pos = synth.grid_positions(w, 957, 3)
    o = torch.empty(w.batch, 3 * T, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    rows = np.arange(0, 3 * T * w.heads, 37)
    ref = np.stack([O.latent_attention(f64(q_c[b]), f64(q_r[b]), q_pos[b].numpy(),
                                       oc.c[b, valid], oc.kr[b, valid], w.head_dim,
                                       spec_of(w)).reshape(-1, w.d_c)[rows]
                    for b in range(w.batch)])
    assert_close(f64(o).reshape(w.batch, -1, w.d_c)[:, rows], ref, what="rollout o_lat")


# ------------------------------------------------------------ edge cases
@pytest.mark.parametrize("d_c", [192, 512])
def test_single_query_token(d_c):
    """Nq = 1: 12 rows in one mostly empty row tile (a lone CTA, or the CTA
    pair of the split-output instance at d_c = 512)."""
    w = small(d_c=d_c, grid_h=6, grid_w=7, window_frames=3, batch=2)
    cache, c, k = upload_cache(w, 61, 3)
    q_c, q_r = synth.draw_queries(w, 1, 62)
    q_pos = synth.grid_positions(w, 2, 1)[:, 5:6].contiguous()
    o = torch.empty(w.batch, 1, w.heads, d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    assert_close(f64(o), oracle_latent(w, q_c, q_r, q_pos, c, k, cache.n_valid()),
                 what=f"Nq=1 d_c={d_c}")


def _chain(w, weights, chunks, q_first, q_n, seed):
    """Append on both sides, then attend with the newest chunk's tokens."""
    cache, oc = run_chunks(w, weights, chunks, seed=seed)
    nq = q_n * w.tokens_per_frame
    q_c, q_r = synth.draw_queries(w, nq, seed + 50)
    q_pos = synth.grid_positions(w, q_first, q_n)
    o = torch.empty(w.batch, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    valid = oc.valid_slots()
    ref = np.stack([O.latent_attention(f64(q_c[b]), f64(q_r[b]), q_pos[b].numpy(),
                                       oc.c[b, valid], oc.kr[b, valid], w.head_dim, spec_of(w))
                    for b in range(w.batch)])
    return f64(o), ref


def test_single_key_window():
    """One token per frame and a one-frame window: a single valid key (the
    rest of its 128-key block masked); the append's token tile holds one
    token and 127 rows past the end."""
    w = small(grid_h=1, grid_w=1, window_frames=1, batch=2)
    weights = synth.draw_layer_weights(w, seed=63)
    got, ref = _chain(w, weights, [(0, 1), (1, 1), (2, 1)], 2, 1, 640)
    assert_close(got, ref, what="single key")


def test_one_frame_window_overwritten():
    """W = 1: every chunk overwrites the whole ring; the current chunk is
    rewritten once more before attention."""
    w = small(grid_h=6, grid_w=6, window_frames=1, batch=2)
    weights = synth.draw_layer_weights(w, seed=65)
    got, ref = _chain(w, weights, [(0, 1), (1, 1), (2, 1), (2, 1)], 2, 1, 660)
    assert_close(got, ref, what="W=1")


def test_positions_at_table_end():
    """Key and query coordinates at the last row of the RoPE table (1023) on
    every axis, next to coordinates at 0."""
    w = small(grid_h=4, grid_w=4, window_frames=2, batch=1)
    assert w.rope_table_len == 1024
    weights = synth.draw_layer_weights(w, seed=67)
    cfg = V.make_config(w)
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    oc = O.OracleCache(w.batch, w.tokens_per_frame, w.window_frames, w.d_c, w.d_r)
    dev = {k: v.cuda() for k, v in weights.items()}
    T = w.tokens_per_frame
    for f in range(2):
        x = synth.draw_tokens(w, T, 680 + f)
        pos = synth.grid_positions(w, f, 1)
        pos[:, :, 0] = 1022 + f
        pos[:, ::2, 1:] = 1023 - pos[:, ::2, 1:]     # half the tokens at the top rows
        V.mla_cache_append(cache, x.cuda(), dev["w_dkv"], dev["gamma_kv"], dev["w_kr"],
                           pos.cuda(), f, 1)
        O.cache_append(oc, f64(x), f64(weights["w_dkv"]), f64(weights["w_kr"]), pos.numpy(),
                       f, 1, gamma=f64(weights["gamma_kv"]), eps=w.rms_eps, spec=spec_of(w))
    q_c, q_r = synth.draw_queries(w, T, 690)
    q_pos = synth.grid_positions(w, 1, 1)
    q_pos[:, :, 0] = 1023
    q_pos[:, 1::2, 1:] = 1023 - q_pos[:, 1::2, 1:]
    o = torch.empty(w.batch, T, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    valid = oc.valid_slots()
    assert_close(f64(cache.c)[:, valid], oc.c[:, valid], what="c at table end")
    assert_close(f64(cache.kr)[:, valid], oc.kr[:, valid], what="k_rope at table end")
    ref = O.latent_attention(f64(q_c[0]), f64(q_r[0]), q_pos[0].numpy(), oc.c[0, valid],
                             oc.kr[0, valid], w.head_dim, spec_of(w))
    assert_close(f64(o)[0], ref, what="attention at table end")


def test_cluster_and_per_tile_append_forms_agree():
    """The Wan chunk at batch 1 takes the cluster form of the append (37
    clusters of 3 CTAs, each 64 columns of c); at batch 2 (222 CTAs would
    exceed one wave) one CTA per token tile computes all 224 columns. The
    same activations give the same cache rows up to one bf16 rounding step
    (the cluster form adds the RMSNorm sum up in three partial sums)."""
    w1 = synth.workload("wan")
    w2 = w1.with_(batch=2)
    weights = {k: v.cuda() for k, v in synth.draw_layer_weights(w1, 69).items()}
    x1 = synth.draw_tokens(w1, w1.chunk_tokens, 70)
    x2 = torch.cat([x1, synth.draw_tokens(w1, w1.chunk_tokens, 71)], 0)
    out = []
    for w, x in ((w1, x1), (w2, x2)):
        cache = V.LatentCache(V.make_config(w))
        V.mla_cache_reset(cache)
        pos = synth.grid_positions(w, 0, w.chunk_frames).cuda()
        V.mla_cache_append(cache, x.cuda(), weights["w_dkv"], weights["gamma_kv"],
                           weights["w_kr"], pos, 0, w.chunk_frames)
        torch.cuda.synchronize()
        n = w.chunk_tokens
        out.append((cache.c[0, :n].float().cpu(), cache.kr[0, :n].float().cpu()))
    (c1, k1), (c2, k2) = out
    for a, b_, name in ((c1, c2, "c"), (k1, k2, "k^R")):
        assert torch.all((a - b_).abs() <= 2.0 ** -7 * b_.abs() + 1e-6), f"{name}: beyond 1 ulp"
    # and both against the oracle on sampled tokens
    rows = np.random.default_rng(2).choice(w1.chunk_tokens, 24, replace=False)
    xs = f64(x1)[0, rows]
    pos = synth.grid_positions(w1, 0, w1.chunk_frames)[0, rows].numpy()
    oc = O.OracleCache(1, len(rows), 1, w1.d_c, w1.d_r)
    O.cache_append(oc, xs[None], f64(weights["w_dkv"].cpu()), f64(weights["w_kr"].cpu()), pos[None],
                   0, 1, gamma=f64(weights["gamma_kv"].cpu()), eps=w1.rms_eps, spec=spec_of(w1))
    assert_close(c1.numpy()[rows], oc.c[0], what="cluster-form c")
    assert_close(k1.numpy()[rows], oc.kr[0], what="cluster-form k_rope")


def test_two_ctas_per_sm_append_form_is_bit_identical():
    """At batch 4 the Wan chunk's 148 token tiles fill one wave, one CTA per
    SM; at batch 5 (185 tiles) two CTAs share each SM with fewer pipeline
    stages. Both run the same MMAs in the same K order, so the four batch
    elements they share come out bit-identical (ragged last tile included);
    the fifth is checked against the oracle on sampled tokens."""
    w4 = synth.workload("wan", batch=4)
    w5 = w4.with_(batch=5)
    weights = {k: v.cuda() for k, v in synth.draw_layer_weights(w4, 72).items()}
    x5 = synth.draw_tokens(w5, w5.chunk_tokens, 73)
    out = []
    for w, x in ((w4, x5[:4]), (w5, x5)):
        cache = V.LatentCache(V.make_config(w))
        V.mla_cache_reset(cache)
        pos = synth.grid_positions(w, 0, w.chunk_frames).cuda()
        V.mla_cache_append(cache, x.contiguous().cuda(), weights["w_dkv"], weights["gamma_kv"],
                           weights["w_kr"], pos, 0, w.chunk_frames)
        torch.cuda.synchronize()
        n = w.chunk_tokens
        out.append((cache.c[:, :n].cpu(), cache.kr[:, :n].cpu()))
    (c4, k4), (c5, k5) = out
    assert torch.equal(c4, c5[:4]) and torch.equal(k4, k5[:4])
    rows = np.concatenate([np.random.default_rng(3).choice(w4.chunk_tokens - 72, 20, replace=False),
                           w4.chunk_tokens - 1 - np.arange(4)])  # + the ragged tile's last rows
    xs = f64(x5)[4, rows]
    pos = synth.grid_positions(w4, 0, w4.chunk_frames)[0, rows].numpy()
    oc = O.OracleCache(1, len(rows), 1, w4.d_c, w4.d_r)
    O.cache_append(oc, xs[None], f64(weights["w_dkv"].cpu()), f64(weights["w_kr"].cpu()), pos[None],
                   0, 1, gamma=f64(weights["gamma_kv"].cpu()), eps=w4.rms_eps, spec=spec_of(w4))
    assert_close(f64(c5[4, rows]), oc.c[0], what="two-per-SM form c")
    assert_close(f64(k5[4, rows]), oc.kr[0], what="two-per-SM form k_rope")


# ------------------------------------------------------------ error paths
def test_position_out_of_table_sets_device_status():
    w = small()
    cfg = V.make_config(w)
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    weights = {k: v.cuda() for k, v in synth.draw_layer_weights(w, 3).items()}
    x = synth.draw_tokens(w, w.tokens_per_frame, 4).cuda()
    pos = synth.grid_positions(w, 0, 1).cuda()
    pos[0, 5, 0] = w.rope_table_len          # one coordinate past the table
    V.mla_cache_append(cache, x, weights["w_dkv"], weights["gamma_kv"], weights["w_kr"], pos, 0, 1)
    assert V.mla_device_status(clear=True) == V.MLA_ERR_RANGE
    assert V.mla_device_status(clear=True) == V.MLA_OK


def test_host_argument_errors():
    w = small()
    cfg = V.make_config(w)
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    q_c, q_r = synth.draw_queries(w, 8, 1)
    q_pos = synth.grid_positions(w, 0, 1)[:, :8].contiguous()
    o = torch.empty(1, 8, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(V.MlaError) as e:       # empty window
        V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    assert e.value.code == V.MLA_ERR_ARG
    weights = {k: v.cuda() for k, v in synth.draw_layer_weights(w, 3).items()}
    x = synth.draw_tokens(w, w.tokens_per_frame, 4).cuda()
    pos = synth.grid_positions(w, 2, 1).cuda()
    with pytest.raises(V.MlaError) as e:       # a gap: frame 2 before frames 0, 1
        V.mla_cache_append(cache, x, weights["w_dkv"], None, weights["w_kr"], pos, 2, 1)
    assert e.value.code == V.MLA_ERR_ARG


def test_host_and_pinned_memory_refused():
    """Every buffer must be device memory of the current device: the kernels'
    TMA copies and cluster multicast address this GPU's own memory only. Host
    tensors, pageable or pinned, are refused before anything is enqueued."""
    import ctypes
    w = small()
    cfg = V.make_config(w)
    cache = V.LatentCache(cfg)
    V.mla_cache_reset(cache)
    cache.frames_written = w.window_frames
    q_c, q_r = synth.draw_queries(w, 8, 1)
    q_pos = synth.grid_positions(w, 0, 1)[:, :8].contiguous()
    o = torch.empty(1, 8, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    lib = V.load()
    dev = [q_c.cuda(), q_r.cuda(), q_pos.cuda()]
    for host in (q_c.clone(), q_c.pin_memory()):
        args = [host, dev[1], dev[2]]
        rc = lib.mla_attention_forward(ctypes.byref(cache.struct),
                                       *[ctypes.c_void_p(t.data_ptr()) for t in args], 8,
                                       ctypes.c_void_p(o.data_ptr()), None)
        assert rc == V.MLA_ERR_ARG
    o_host = torch.empty(o.shape, dtype=o.dtype).pin_memory()
    rc = lib.mla_attention_forward(ctypes.byref(cache.struct),
                                   *[ctypes.c_void_p(t.data_ptr()) for t in dev], 8,
                                   ctypes.c_void_p(o_host.data_ptr()), None)
    assert rc == V.MLA_ERR_ARG
    V.mla_attention_forward(cache, *dev, o)           # the same call on device memory runs
    torch.cuda.synchronize()


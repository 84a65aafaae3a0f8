"""mla_attention_forward_ws: the absorbed attention with the last, partial wave
of row tiles split over the SMs by key range (pieces of a tile combined by
the last to finish: the online softmax of Eq. score split over keys, App. E's
latent output). Checked through the C ABI against the float64 oracle on rows
of the split tiles and of the whole tiles, row by row, and against the
unsplit entry point on every row."""

import ctypes

import numpy as np
import pytest
import torch

from oracle import mla_oracle as O
from paper_2605_30351_gb300 import synth
from paper_2605_30351_gb300 import videomla as V

from test_gpu_parity import assert_close, assert_rows_close, f64, spec_of
from test_gpu_softmax import absorbed_inputs, oracle_absorbed_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    V.load()
    V.mla_device_status(clear=True)
    yield
    assert V.mla_device_status(clear=True) == V.MLA_OK


def sms():
    return torch.cuda.get_device_properties(0).multi_processor_count


def split_rows(w, nq):
    """First row of the tiles that the split covers (pairs of 128-row tiles
    beyond the last whole wave of SMs/2 pairs), or None when nothing is split."""
    tiles = -(-nq * w.heads // 128)
    pairs = -(-tiles // 2)
    total = pairs * w.batch
    slots = sms() // 2
    full, rest = divmod(total, slots)
    if full < 1 or rest < 1:
        return None
    first_pair = full * slots            # global pair index (b * pairs + pair)
    return first_pair // pairs, (first_pair % pairs) * 256


def run_both(w, q_c, q_r, q_pos, c, k):
    cache = V.LatentCache(V.make_config(w))
    cache.c.copy_(c)
    cache.kr.copy_(k)
    cache.frames_written = w.window_frames
    nq = q_c.shape[1]
    args = (q_c.cuda(), q_r.cuda(), q_pos.cuda())
    o_ws = torch.empty(w.batch, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(V.mla_attention_workspace_bytes(cache.cfg, nq), dtype=torch.uint8,
                     device="cuda")
    V.mla_attention_forward_ws(cache, *args, ws, o_ws)
    o = torch.empty_like(o_ws)
    V.mla_attention_forward(cache, *args, o)
    torch.cuda.synchronize()
    rs = lambda t: f64(t).reshape(w.batch, nq * w.heads, w.d_c)
    return rs(o_ws), rs(o)


def check(w, nq, case, seed, extra=48):
    q_c, q_r, c, k, _ = absorbed_inputs(w, nq, case, seed)
    ff = w.window_frames - w.chunk_frames
    q_pos = synth.grid_positions(w, ff, w.chunk_frames)[:, :nq].contiguous()
    got, plain = run_both(w, q_c, q_r, q_pos, c, k)
    # every row: the split and the unsplit kernel agree
    assert_rows_close(got.reshape(-1, w.d_c), plain.reshape(-1, w.d_c), f"{case}: ws vs plain")
    sp = split_rows(w, nq)
    assert sp is not None, "the shape must leave a partial last wave"
    b_sp, row_sp = sp
    n_rows = nq * w.heads
    rng = np.random.default_rng(seed)
    for b in range(w.batch):
        lo = row_sp if b == b_sp else (0 if b > b_sp else n_rows)
        rows = [0, 1, 127, 128, n_rows - 1]
        if lo < n_rows:  # rows of split tiles: both CTAs of a pair, tile edges
            rows += [lo, lo + 1, lo + 127, lo + 128, lo + 255, (lo + n_rows) // 2]
            rows += list(rng.integers(lo, n_rows, extra))
        rows += list(rng.integers(0, n_rows, extra // 4))
        rows = np.unique(np.asarray([x for x in rows if 0 <= x < n_rows]))
        ref, _ = oracle_absorbed_rows(w, q_c, q_r, q_pos, c, k, b, rows)
        assert_rows_close(got[b, rows], ref, f"{case} b={b} (split from row {lo})")


@pytest.mark.parametrize("case", ["plain", "late", "early", "mixture"])
def test_split_wan_shape(case):
    """The Wan-1.3B layer shape: 220 tile pairs, two whole waves of SMs/2 and
    68 pairs whose 256 key blocks are shared by every pair of the last wave.
    The late, early and mixture cases give the pieces of a tile running maxima
    far apart, which the combine must weigh."""
    w = synth.workload("wan")
    if case == "plain":
        q_c, q_r = synth.draw_queries(w, w.chunk_tokens, 1100)
        c, k = synth.draw_cache_rows(w, w.slots, 1101)
        q_pos = synth.grid_positions(w, 18, 3)
        got, plain = run_both(w, q_c, q_r, q_pos, c, k)
        assert_rows_close(got.reshape(-1, w.d_c), plain.reshape(-1, w.d_c), "ws vs plain")
        lo = split_rows(w, w.chunk_tokens)[1]
        rows = np.unique(np.concatenate([[0, lo, lo + 1, lo + 128, 56159],
                                         np.random.default_rng(3).integers(lo, 56160, 60)]))
        ref, _ = oracle_absorbed_rows(w, q_c, q_r, q_pos, c, k, 0, rows)
        assert_rows_close(got[0, rows], ref, "wan split rows")
    else:
        check(w, w.chunk_tokens, case, 1110 + len(case))


def test_split_rollout_batch4():
    """Batch 4 (880 tile pairs: 11 whole waves, the last 44 pairs split, all in
    the last batch element)."""
    w = synth.workload("wan", batch=4)
    check(w, w.chunk_tokens, "late", 1120, extra=24)


@pytest.mark.parametrize("d_c,d_r,pairs,dims", [
    (64, 32, (6, 5, 5), (44, 42, 42)), (128, 64, (12, 10, 10), (64, 64, 64)),
    (192, 64, (12, 10, 10), (64, 64, 64)),
])
def test_split_other_latent_sizes(d_c, d_r, pairs, dims):
    w = synth.workload("wan", d_c=d_c, d_r=d_r, rope_pairs=pairs, rope_axis_dims=dims)
    check(w, w.chunk_tokens, "mixture", 1130 + d_c + d_r, extra=24)


def test_split_short_window_many_slots():
    """1700 tokens (160 row tiles, 80 pairs: one whole wave and 4 split pairs)
    against a window of 2 frames of 65 tokens (130 keys: two key blocks, the
    second ragged): 8 slots of one key block each, two pieces per tile."""
    w = synth.workload("tiny", grid_h=5, grid_w=13, window_frames=2, chunk_frames=1, batch=1,
                       rope_pairs=(6, 5, 5))
    nq = 1700
    q_c, q_r, c, k, _ = absorbed_inputs(w, nq, "late", 1140)
    q_pos = torch.zeros(1, nq, 3, dtype=torch.int32)
    q_pos[0, :, 0] = 1
    q_pos[0, :, 1] = torch.arange(nq) % 5
    q_pos[0, :, 2] = torch.arange(nq) % 13
    got, plain = run_both(w, q_c, q_r, q_pos, c, k)
    assert_rows_close(got.reshape(-1, w.d_c), plain.reshape(-1, w.d_c), "ws vs plain")
    rows = np.arange(nq * w.heads)
    ref, _ = oracle_absorbed_rows(w, q_c, q_r, q_pos, c, k, 0, rows)
    assert_rows_close(got[0], ref, "short window, every row")


def test_split_workspace_rules():
    w = synth.workload("wan")
    cfg = V.make_config(w)
    need = V.mla_attention_workspace_bytes(cfg, w.chunk_tokens)
    slots = sms() // 2
    assert need >= slots * 2 * 2 * 128 * w.d_c * 4
    cache = V.LatentCache(cfg)
    cache.frames_written = w.window_frames
    q_c = torch.zeros(1, w.chunk_tokens, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    q_r = torch.zeros(1, w.chunk_tokens, w.heads, w.d_r, dtype=torch.bfloat16, device="cuda")
    q_pos = torch.zeros(1, w.chunk_tokens, 3, dtype=torch.int32, device="cuda")
    o = torch.empty_like(q_c)
    small = torch.empty(need - 256, dtype=torch.uint8, device="cuda")
    with pytest.raises(V.MlaError) as e:
        V.mla_attention_forward_ws(cache, q_c, q_r, q_pos, small, o)
    assert e.value.code == V.MLA_ERR_ARG
    host_ws = torch.empty(need, dtype=torch.uint8).pin_memory()
    lib = V.load()
    rc = lib.mla_attention_forward_ws(ctypes.byref(cache.struct), ctypes.c_void_p(q_c.data_ptr()),
                                      ctypes.c_void_p(q_r.data_ptr()),
                                      ctypes.c_void_p(q_pos.data_ptr()), w.chunk_tokens,
                                      ctypes.c_void_p(host_ws.data_ptr()), need,
                                      ctypes.c_void_p(o.data_ptr()), None)
    assert rc == V.MLA_ERR_ARG
    # a call that is too small to leave a partial wave runs unsplit
    nq = 100
    got = torch.empty(1, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    V.mla_attention_forward_ws(cache, q_c[:, :nq].contiguous(), q_r[:, :nq].contiguous(),
                               q_pos[:, :nq].contiguous(), ws, got)
    torch.cuda.synchronize()
    # zero queries: every score 0, the output is the mean latent (the cache is zero)
    assert float(got.float().abs().max()) == 0.0

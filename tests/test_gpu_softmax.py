"""The online softmax's hard cases (Eq. score and the softmax over the window,
Sec. 3.3), for the absorbed kernel and the dense baseline, through the C ABI,
against the float64 oracle, checked row by row.

With the default synthetic inputs every score has unit variance, so a row's
running maximum never grows past the kernels' lazy-rescale margin (2^8 in
log2 units) after its first key block and the output rescale never runs.
These inputs are built so that it must, and so that the rows that rescale
share warps with rows that do not:
  peaked    content queries scaled so the scores have standard deviation 12
  late      one key in the LAST key block aligned with the queries of a third
            of the rows, ~60 above their other scores: the running maximum
            jumps far past the margin at the last block (near one-hot rows)
  early     the same key in the FIRST block: every later block lies far
            below the running maximum (its exponentials underflow to zero)
  mixture   a key in the last block holding about half of its rows' softmax
            mass (unit-variance scores otherwise), so the rescale factor
            decides half of the output (windows of >= 4000 keys)
  uniform   a third of the rows with zero queries: every score is 0 and the
            output is the mean of the valid latents
For the late and mixture cases the test also checks, from the oracle's
probabilities, that the planted rows' running maximum crosses the margin
(so the kernel's rescale branch runs for them); the debug build counts the
rescales it performs (tests/test_gpu_debug_build.py).

Checks: every sampled row has relative L2 error <= 1e-2 and max-abs error
<= 1e-2 of that row's largest |reference| value; over all rows, max-abs
<= 2e-2 and relative L2 <= 1e-2. Sampled rows cover the first, second (the
other CTA of the first pair), a middle and the last row tile."""

import math

import numpy as np
import pytest
import torch

from oracle import mla_oracle as O
from paper_2605_30351_gb300 import synth
from paper_2605_30351_gb300 import videomla as V

from test_gpu_parity import assert_rows_close, f64, spec_of

pytestmark = pytest.mark.gpu

MARGIN_LOG2 = 8.0      # lazy-rescale margin of the tensor-core kernels
KEY_BLOCK = 128        # keys per block (d_c <= 256 and the dense kernel)
CASES = ("peaked", "late", "early", "mixture", "uniform")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    V.load()
    V.mla_device_status(clear=True)
    yield
    assert V.mla_device_status(clear=True) == V.MLA_OK


def rescale_events(logp, n_valid):
    """Rescales the kernels' lazy rule performs for one row, from the row's
    natural-log probabilities over the valid keys (score differences): the
    running maximum starts at the first block's maximum and moves only when a
    later block's maximum exceeds it by more than MARGIN_LOG2 (log2 units)."""
    s = np.asarray(logp, dtype=np.float64) * math.log2(math.e)
    m_run = None
    events = 0
    for j0 in range(0, n_valid, KEY_BLOCK):
        m_blk = np.max(s[j0:j0 + KEY_BLOCK])
        if m_run is None:
            m_run = m_blk
        elif m_blk > m_run + MARGIN_LOG2:
            events += 1
            m_run = m_blk
    return events


def planted_rows(n_rows):
    return np.arange(n_rows) % 3 == 0


# -------------------------------------------------------- absorbed form
def absorbed_inputs(w, nq, case, seed):
    """q_c, q_r, cache rows c, k (bf16) with the case's structure; rows are
    (token, head) pairs, a third of them planted. Returns the planted mask too."""
    B, H, dc = w.batch, w.heads, w.d_c
    n_valid = w.slots
    q_c, q_r = synth.draw_queries(w, nq, seed, as_float64=True)
    c, k = synth.draw_cache_rows(w, w.slots, seed + 1, as_float64=True)
    rows = nq * H
    sel = planted_rows(rows).reshape(nq, H)
    qc_flat = q_c.reshape(B, rows, dc)
    if case == "peaked":
        q_c = q_c * (12.0 * math.sqrt(w.head_dim / dc) / q_c.std())
    elif case in ("late", "early", "mixture"):
        j_star = n_valid - 3 if case != "early" else 5
        u = synth.unit_vectors(B, dc, seed + 2)
        # the planted key: a latent of the same norm as the others, along u
        c[:, j_star] = u * math.sqrt(dc)
        # its score for a planted row rises by beta |c*| / sqrt(head_dim)
        target = 60.0 if case != "mixture" else math.log(n_valid) + 0.5
        beta = target * math.sqrt(w.head_dim) / math.sqrt(dc)
        qc_flat[:, sel.reshape(-1)] += beta * u[:, None, :]
        q_c = qc_flat.reshape(B, nq, H, dc)
    elif case == "uniform":
        q_c[:, sel] = 0.0
        q_r[:, sel] = 0.0
    return (synth.bf16(q_c), synth.bf16(q_r), synth.bf16(c), synth.bf16(k),
            sel.reshape(-1))


def run_absorbed(w, q_c, q_r, c, k, q_pos, flags=0):
    cache = V.LatentCache(V.make_config(w, flags))
    cache.c.copy_(c)
    cache.kr.copy_(k)
    cache.frames_written = w.window_frames
    nq = q_c.shape[1]
    o = torch.empty(w.batch, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos.cuda(), o)
    torch.cuda.synchronize()
    return f64(o).reshape(w.batch, nq * w.heads, w.d_c)


def oracle_absorbed_rows(w, q_c, q_r, q_pos, c, k, b, rows):
    """Oracle output and probabilities of (token, head) rows of batch element
    b: each row is passed as a one-head query at its token's position."""
    tok, head = rows // w.heads, rows % w.heads
    qc = f64(q_c[b])[tok, head][:, None]
    qr = f64(q_r[b])[tok, head][:, None]
    o, p = O.latent_attention(qc, qr, q_pos[b].numpy()[tok], f64(c[b]), f64(k[b]), w.head_dim,
                              spec_of(w), return_probs=True)
    return o[:, 0], p[:, 0]


def sample_rows(n_rows, extra, seed):
    """Rows of the first two row tiles (both CTAs of the first pair), a middle
    and the last tile, plus `extra` random rows."""
    rng = np.random.default_rng(seed)
    fixed = [0, 1, 2, 30, 31, 32, 33, 63, 64, 95, 96, 127, 128, 129, 130, 200, 255,
             n_rows // 2, n_rows // 2 + 1, n_rows - 3, n_rows - 2, n_rows - 1]
    rows = np.concatenate([fixed, rng.choice(n_rows, extra, replace=False)])
    return np.unique(rows[rows < n_rows])


def check_absorbed(w, nq, case, seed, flags=0, extra=40, first_frame=None):
    q_c, q_r, c, k, sel = absorbed_inputs(w, nq, case, seed)
    ff = w.window_frames - w.chunk_frames if first_frame is None else first_frame
    q_pos = synth.grid_positions(w, ff, w.chunk_frames)[:, :nq].contiguous()
    got = run_absorbed(w, q_c, q_r, c, k, q_pos, flags)
    n_rows = nq * w.heads
    for b in range(w.batch):
        rows = sample_rows(n_rows, min(extra, n_rows), seed + b)
        ref, p = oracle_absorbed_rows(w, q_c, q_r, q_pos, c, k, b, rows)
        assert_rows_close(got[b, rows], ref, f"{case} b={b}")
        if case in ("late", "mixture"):
            with np.errstate(divide="ignore"):
                ev = [rescale_events(np.log(p[i]), w.slots) for i in range(len(rows))
                      if sel[rows[i]]]
            assert ev and np.mean(np.asarray(ev) > 0) >= 0.75, ev
        if case in ("late", "early"):
            j_star = w.slots - 3 if case == "late" else 5
            planted = sel[rows]
            # near one-hot: the planted key carries (almost) all of the mass
            assert np.all(p[planted, j_star] > 1 - 1e-6)
        if case == "mixture":
            mass = p[sel[rows], w.slots - 3]
            assert 0.2 < np.median(mass) < 0.8, np.median(mass)
        if case == "uniform":
            flat = p[sel[rows]]
            assert np.allclose(flat, 1.0 / w.slots, rtol=1e-12)


@pytest.mark.parametrize("flags", [0, V.MLA_FLAG_SIMT])
@pytest.mark.parametrize("case", ("peaked", "late", "early", "uniform"))
def test_absorbed_hard_cases_small(case, flags):
    """390 keys (three full key blocks and a 6-key ragged one), 480 rows
    (a ragged fourth row tile), batch 2."""
    w = synth.workload("tiny", grid_h=10, grid_w=13, window_frames=3, batch=2,
                       rope_pairs=(6, 5, 5))
    check_absorbed(w, 40, case, 910 + CASES.index(case), flags, first_frame=2)


@pytest.mark.parametrize("case", CASES)
def test_absorbed_hard_cases_full_window(case):
    """The full 21-frame Wan window (32,760 keys: 256 key blocks, the last
    ragged) against a 40-token chunk (480 rows), every row checked."""
    w = synth.workload("wan", chunk_frames=1)
    q_c, q_r, c, k, sel = absorbed_inputs(w, 40, case, 930 + CASES.index(case))
    q_pos = synth.grid_positions(w, 20, 1)[:, :40].contiguous()
    got = run_absorbed(w, q_c, q_r, c, k, q_pos)
    rows = np.arange(480)
    ref, p = oracle_absorbed_rows(w, q_c, q_r, q_pos, c, k, 0, rows)
    assert_rows_close(got[0], ref, f"{case} full window")
    if case in ("late", "mixture"):
        with np.errstate(divide="ignore"):
            ev = np.array([rescale_events(np.log(p[i]), w.slots) for i in rows[sel]])
        assert np.mean(ev > 0) >= 0.75, ev


@pytest.mark.parametrize("case", CASES)
def test_absorbed_hard_cases_wan_shape(case):
    """The Wan-1.3B layer shape (4680 x 12 rows, 32,760 keys) on sampled rows."""
    w = synth.workload("wan")
    check_absorbed(w, w.chunk_tokens, case, 950 + CASES.index(case), extra=60)


@pytest.mark.parametrize("d_c,d_r,pairs,dims", [
    (64, 32, (6, 5, 5), (44, 42, 42)), (256, 64, (12, 10, 10), (64, 64, 64)),
])
def test_absorbed_late_key_other_latent_sizes(d_c, d_r, pairs, dims):
    """Q in TMEM (d_c = 64) and Q split between TMEM and shared memory
    ((256, 64)): the late dominant key at the full window."""
    w = synth.workload("wan", chunk_frames=1, d_c=d_c, d_r=d_r, rope_pairs=pairs,
                       rope_axis_dims=dims)
    check_absorbed(w, 40, "late", 970 + d_c, extra=480)


@pytest.mark.parametrize("case", ("late", "mixture"))
def test_absorbed_hard_cases_dc512(case):
    """d_c = 512 (64-key blocks; both CTAs of a pair run the same softmax on
    the same scores and each rescales its half of the output)."""
    w = synth.workload("wan", chunk_frames=1, d_c=512)
    q_c, q_r, c, k, sel = absorbed_inputs(w, 40, case, 980 + CASES.index(case))
    q_pos = synth.grid_positions(w, 20, 1)[:, :40].contiguous()
    got = run_absorbed(w, q_c, q_r, c, k, q_pos)
    rows = sample_rows(480, 120, 5)
    ref, _ = oracle_absorbed_rows(w, q_c, q_r, q_pos, c, k, 0, rows)
    assert_rows_close(got[0, rows], ref, f"{case} d_c=512")


# ----------------------------------------------------------- dense baseline
def dense_inputs(w, nq, slots, case, seed):
    """q [B, nq, H, d_h], k, v [B, H, slots, d_h] (bf16) with the case's
    structure; rows are tokens of each head, a third of them planted."""
    rng = np.random.default_rng(seed)
    B, H, dh = w.batch, w.heads, w.head_dim
    q = rng.standard_normal((B, nq, H, dh))
    k = rng.standard_normal((B, H, slots, dh))
    v = rng.standard_normal((B, H, slots, dh))
    sel = planted_rows(nq)
    if case == "peaked":
        q *= 12.0
    elif case in ("late", "early", "mixture"):
        j_star = slots - 3 if case != "early" else 5
        u = synth.unit_vectors(B * H, dh, seed + 1).reshape(B, H, dh)
        k[:, :, j_star] = u * math.sqrt(dh)
        target = 60.0 if case != "mixture" else math.log(slots) + 0.5
        q[:, sel] += target * u[:, None, :, :]
    elif case == "uniform":
        q[:, sel] = 0.0
    return synth.bf16(q), synth.bf16(k), synth.bf16(v), sel


def check_dense(w, nq, slots, case, seed, tokens):
    q, k, v, sel = dense_inputs(w, nq, slots, case, seed)
    o = torch.empty(q.shape, dtype=torch.bfloat16, device="cuda")
    V.mla_dense_attention_forward(V.make_config(w), q.cuda(), k.cuda(), v.cuda(), slots, o)
    torch.cuda.synchronize()
    got = f64(o)
    for b in range(w.batch):
        ref, p = O.dense_attention(f64(q[b, tokens]), f64(k[b]), f64(v[b]), w.head_dim,
                                   return_probs=True)
        assert_rows_close(got[b, tokens], ref, f"dense {case} b={b}")
        if case in ("late", "mixture"):
            with np.errstate(divide="ignore"):
                ev = [rescale_events(np.log(p[i, h]), slots)
                      for i in range(len(tokens)) if sel[tokens[i]] for h in range(w.heads)]
            assert ev and np.mean(np.asarray(ev) > 0) >= 0.75
        if case == "uniform":
            assert np.allclose(p[sel[tokens]], 1.0 / slots, rtol=1e-12)


@pytest.mark.parametrize("case", ("peaked", "late", "early", "uniform"))
def test_dense_hard_cases_small(case):
    """300 tokens (a ragged third row tile) x 12 heads against 500 keys, batch 2."""
    w = synth.workload("tiny", batch=2)
    check_dense(w, 300, 500, case, 990 + CASES.index(case), np.arange(300))


@pytest.mark.parametrize("case", CASES)
def test_dense_hard_cases_wan_shape(case):
    """The dense baseline at the Wan shape (4680 tokens x 12 heads, 32,760 keys)
    on sampled tokens of the first, second, a middle and the last row tile."""
    w = synth.workload("wan")
    n = w.chunk_tokens
    tokens = np.unique(np.concatenate([[0, 1, 2, 3, 64, 127, 128, 129, 255, n // 2, n - 2, n - 1],
                                       np.random.default_rng(7).choice(n, 24, replace=False)]))
    check_dense(w, n, w.slots, case, 1000 + CASES.index(case), tokens)

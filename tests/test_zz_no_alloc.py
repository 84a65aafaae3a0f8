"""The allocation-free query prologue (mla_query_prologue_noalloc).

Some callers cannot allocate device memory when they run the layer (inside
another framework's memory pool, or in a real-time loop where cudaMalloc and
cudaFree are not allowed), so this entry point keeps its intermediate buffer
in a fixed array inside the library instead of taking a workspace. These
tests call it through the C ABI and check it against the regular entry point
(which uses a caller-provided workspace) on two calls in a row, and check that
a request larger than the fixed array is refused before any work is queued.

The file name makes pytest collect it last."""

import ctypes

import pytest
import torch

from paper_2605_30351_gb300 import synth
from paper_2605_30351_gb300 import videomla as V

from test_gpu_parity import assert_close, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def layer():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    V.load()
    w = synth.workload("wan")                        # one Wan-1.3B chunk: 4680 query tokens
    cfg = V.make_config(w)
    wt = {k: v.cuda() for k, v in synth.draw_layer_weights(w, seed=301).items()}
    w_qcat, _ = V.mla_absorb_weights(cfg, wt["w_uq"], wt["w_uk"], wt["w_qr"], wt["gamma_q"],
                                     wt["w_uv"], wt["w_o"])
    return w, cfg, wt, w_qcat


def _outputs(w, nq):
    shape_c = (w.batch, nq, w.heads, w.d_c)
    shape_r = (w.batch, nq, w.heads, w.d_r)
    return (torch.empty(shape_c, dtype=torch.bfloat16, device="cuda"),
            torch.empty(shape_r, dtype=torch.bfloat16, device="cuda"))


def test_noalloc_matches_workspace_entry_point_twice(layer):
    w, cfg, wt, w_qcat = layer
    nq = w.chunk_tokens
    assert V.mla_query_workspace_bytes(cfg, nq) <= V.MLA_NOALLOC_SCRATCH_BYTES
    ws = torch.empty(V.mla_query_workspace_bytes(cfg, nq), dtype=torch.uint8, device="cuda")
    for call, seed in enumerate((302, 303)):        # the second call reuses the dirty array
        x = synth.draw_tokens(w, nq, seed).cuda()
        ref_c, ref_r = _outputs(w, nq)
        V.mla_query_prologue(cfg, x, wt["w_dq"], w_qcat, ws, ref_c, ref_r)
        got_c, got_r = _outputs(w, nq)
        V.mla_query_prologue_noalloc(cfg, x, wt["w_dq"], w_qcat, got_c, got_r)
        torch.cuda.synchronize()
        assert_close(f64(got_c), f64(ref_c), what=f"q_c, call {call}")
        assert_close(f64(got_r), f64(ref_r), what=f"q_r, call {call}")
    assert V.mla_device_status(clear=True) == V.MLA_OK


def test_noalloc_refuses_requests_beyond_its_scratch(layer):
    w, cfg, _wt, _w_qcat = layer
    big = cfg.__class__.from_buffer_copy(cfg)
    big.batch = 2                                    # two chunks need ~14.5 MB > 8 MiB
    assert V.mla_query_workspace_bytes(big, w.chunk_tokens) > V.MLA_NOALLOC_SCRATCH_BYTES
    fake = ctypes.c_void_p(1 << 20)                  # never dereferenced: refused first
    rc = V.load().mla_query_prologue_noalloc(ctypes.byref(big), fake, fake, fake,
                                             w.chunk_tokens, fake, fake, None)
    assert rc == V.MLA_ERR_TOO_LARGE
    assert "no-allocation" in V.load().mla_status_string(rc).decode()


def _compare_twice(w, cfg, wt, w_qcat, nq, seeds):
    ws = torch.empty(V.mla_query_workspace_bytes(cfg, nq), dtype=torch.uint8, device="cuda")
    for call, seed in enumerate(seeds):
        x = synth.draw_tokens(w, nq, seed).cuda()
        ref_c, ref_r = _outputs(w, nq)
        V.mla_query_prologue(cfg, x, wt["w_dq"], w_qcat, ws, ref_c, ref_r)
        got_c, got_r = _outputs(w, nq)
        V.mla_query_prologue_noalloc(cfg, x, wt["w_dq"], w_qcat, got_c, got_r)
        torch.cuda.synchronize()
        assert_close(f64(got_c), f64(ref_c), what=f"q_c, call {call}")
        assert_close(f64(got_r), f64(ref_r), what=f"q_r, call {call}")
    assert V.mla_device_status(clear=True) == V.MLA_OK


def test_noalloc_wide_tiles_match_workspace_entry_point():
    """A query latent of d_q = 128 over five Wan chunks (23,400 rows: 183 row
    tiles) takes the 256-wide first GEMM, whose partial sums of squares use a
    different tile count in the scratch; 6.1 MB still fits the fixed array."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    w = synth.workload("wan", d_q=128, batch=5)
    cfg = V.make_config(w)
    nq = w.chunk_tokens
    need = V.mla_query_workspace_bytes(cfg, nq)
    assert need <= V.MLA_NOALLOC_SCRATCH_BYTES and (w.batch * nq + 127) // 128 >= 152
    wt = {k: v.cuda() for k, v in synth.draw_layer_weights(w, seed=311).items()}
    w_qcat, _ = V.mla_absorb_weights(cfg, wt["w_uq"], wt["w_uk"], wt["w_qr"], wt["gamma_q"],
                                     wt["w_uv"], wt["w_o"])
    _compare_twice(w, cfg, wt, w_qcat, nq, (312, 313))


def test_noalloc_at_the_scratch_limit(layer):
    """The largest query count whose intermediate buffer fits the fixed array
    exactly (d_q = 768: 1552 bytes per token) is accepted and correct; one
    token more is refused before anything is queued."""
    w, cfg, wt, w_qcat = layer
    nq = V.MLA_NOALLOC_SCRATCH_BYTES // 1552
    assert V.mla_query_workspace_bytes(cfg, nq) <= V.MLA_NOALLOC_SCRATCH_BYTES
    assert V.mla_query_workspace_bytes(cfg, nq + 1) > V.MLA_NOALLOC_SCRATCH_BYTES
    _compare_twice(w, cfg, wt, w_qcat, nq, (314, 315))
    x = synth.draw_tokens(w, nq + 1, 316).cuda()
    got_c, got_r = _outputs(w, nq + 1)
    with pytest.raises(V.MlaError) as e:
        V.mla_query_prologue_noalloc(cfg, x, wt["w_dq"], w_qcat, got_c, got_r)
    assert e.value.code == V.MLA_ERR_TOO_LARGE

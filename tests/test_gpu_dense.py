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


@pytest.mark.parametrize("nq,slots,n_valid,batch", [
    (64, 256, 256, 1),     # the tiny config's shape
    (300, 500, 387, 2),    # ragged tiles and a partially valid window
])
def test_dense_attention_matches_oracle(nq, slots, n_valid, batch):
    w = synth.workload("tiny", batch=batch)
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

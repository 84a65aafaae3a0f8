"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every symbol the header declares, validates arguments before any launch, and
its RoPE table matches the oracle's frequencies."""

import ctypes
import os
import re

import numpy as np
import pytest

from oracle import mla_oracle as O
from paper_2605_30351_gb300 import synth
from paper_2605_30351_gb300 import videomla as V

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "videomla.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(mla_[a-z_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol():
    lib = V.load()
    names = declared_functions()
    assert set(names) == set(V.EXPORTS), names
    for n in names:
        assert hasattr(lib, n), n
    assert lib.mla_version() >= 100


def test_struct_layout_matches_header():
    # 12 ints, a double, 4 ints, a float, an unsigned, an int, padded to 8
    assert ctypes.sizeof(V.mla_config) == 88
    assert V.mla_config.rope_theta.offset == 48
    assert V.mla_config.sink_frames.offset == 80
    # three pointers, a long long, the config
    assert ctypes.sizeof(V.mla_cache) == 120
    assert V.mla_cache.cfg.offset == 32


def test_config_validation():
    w = synth.workload("wan")
    cfg = V.make_config(w)
    assert V.mla_config_check(cfg) == V.MLA_OK
    bad = V.make_config(w)
    bad.rope_pairs_t = 7                      # 2*(7+5+5) != 32
    assert V.mla_config_check(bad) == V.MLA_ERR_ARG
    bad = V.make_config(w)
    bad.d_c = 100                             # rows not 16-byte multiples
    assert V.mla_config_check(bad) == V.MLA_ERR_ARG
    bad = V.make_config(w)
    bad.rope_dim_h = 4                        # band width narrower than its pairs
    assert V.mla_config_check(bad) == V.MLA_ERR_ARG
    bad = V.make_config(w)
    bad.window_frames = 0
    assert V.mla_config_check(bad) == V.MLA_ERR_ARG
    bad = V.make_config(w)
    bad.d_r = 0                               # no positional key (and no RoPE pairs)
    bad.rope_pairs_t = bad.rope_pairs_h = bad.rope_pairs_w = 0
    assert V.mla_config_check(bad) == V.MLA_ERR_ARG
    bad = V.make_config(w)
    bad.sink_frames = w.window_frames         # no frame slot left for the FIFO part
    assert V.mla_config_check(bad) == V.MLA_ERR_ARG
    bad.sink_frames = -1
    assert V.mla_config_check(bad) == V.MLA_ERR_ARG
    sink = V.make_config(synth.workload("sink"))
    assert V.mla_config_check(sink) == V.MLA_OK
    assert sink.sink_frames == 1 and sink.flags & V.MLA_FLAG_ROTATE_AT_USE


def test_window_path_argument_rules():
    """Rotate-at-use caches must go through the window entry point and vice
    versa; the window workspace is sized for keys plus query positions."""
    lib = V.load()
    fake = ctypes.c_void_p(1 << 20)
    w = synth.workload("sink")
    cfg = V.make_config(w)
    cache = V.mla_cache(c=fake, kr=fake, rope_table=fake, frames_written=9, cfg=cfg)
    assert lib.mla_attention_forward(ctypes.byref(cache), fake, fake, fake, 4680, fake,
                                     None) == V.MLA_ERR_ARG
    need = V.mla_window_workspace_bytes(cfg, 4680)
    keys = w.batch * w.slots * w.d_r * 2
    assert need == (keys + 255) // 256 * 256 + w.batch * 4680 * 12
    assert lib.mla_attention_window_forward(ctypes.byref(cache), fake, fake, fake, 4680, fake,
                                            fake, need - 1, fake, None) == V.MLA_ERR_ARG
    plain = V.mla_cache(c=fake, kr=fake, rope_table=fake, frames_written=21,
                        cfg=V.make_config(synth.workload("wan")))
    assert lib.mla_attention_window_forward(ctypes.byref(plain), fake, fake, fake, 4680, fake,
                                            fake, need, fake, None) == V.MLA_ERR_ARG
    # a rotate-at-use append does not need positions: NULL pos passes the
    # host checks up to the frame-range rule
    assert lib.mla_cache_append(ctypes.byref(cache), fake, fake, None, fake, None, 0,
                                w.window_frames + 1, None) == V.MLA_ERR_RANGE


def test_null_arguments_rejected_before_launch():
    lib = V.load()
    w = synth.workload("tiny")
    cache = V.mla_cache(cfg=V.make_config(w))
    assert lib.mla_cache_append(ctypes.byref(cache), None, None, None, None, None, 0, 1,
                                None) == V.MLA_ERR_ARG
    assert lib.mla_attention_forward(ctypes.byref(cache), None, None, None, 1, None,
                                     None) == V.MLA_ERR_ARG
    assert lib.mla_cache_reset(None, None) == V.MLA_ERR_ARG
    # n_frames beyond the window is a range error (checked before pointers are used)
    fake = ctypes.c_void_p(1 << 20)
    cache = V.mla_cache(c=fake, kr=fake, rope_table=fake, cfg=V.make_config(w))
    assert lib.mla_cache_append(ctypes.byref(cache), fake, fake, None, fake, fake, 0,
                                w.window_frames + 1, None) == V.MLA_ERR_RANGE
    # misaligned pointer
    odd = ctypes.c_void_p((1 << 20) + 2)
    assert lib.mla_cache_append(ctypes.byref(cache), odd, fake, None, fake, fake, 0, 1,
                                None) == V.MLA_ERR_ARG
    assert lib.mla_status_string(V.MLA_ERR_RANGE).decode().startswith("frame count")
    # the wait self-test checks its limit before launching anything
    assert lib.mla_selftest_bounded_wait(0, None) == V.MLA_ERR_ARG
    assert lib.mla_selftest_bounded_wait(3_000_000_000, None) == V.MLA_ERR_ARG


@pytest.mark.parametrize("name", ["tiny", "wan"])
def test_rope_table_matches_oracle_frequencies(name):
    w = synth.workload(name)
    tab = V.mla_rope_table_fill(V.make_config(w))
    assert tab.shape == (w.rope_table_len, w.d_r // 2, 2)
    inv, _axis = O.rope_inv_freq(O.RopeSpec(w.rope_pairs, w.rope_axis_dims, w.rope_theta))
    pos = np.arange(w.rope_table_len)[:, None]
    np.testing.assert_allclose(tab[..., 0], np.cos(pos * inv), rtol=0, atol=2e-7)
    np.testing.assert_allclose(tab[..., 1], np.sin(pos * inv), rtol=0, atol=2e-7)


def test_sink_append_takes_at_most_the_fifo_slots():
    """Frames past the S sinks share W - S frame slots (App. D.4), so one
    append may carry at most W - S of them: a longer run would write two
    frames to the same slots. The rule is checked on the host, before any
    pointer is used (the later residency check then fails on fake pointers,
    with MLA_ERR_ARG on a GPU machine or MLA_ERR_CUDA without a device)."""
    lib = V.load()
    fake = ctypes.c_void_p(1 << 20)

    def append(w, first, n, written):
        cache = V.mla_cache(c=fake, kr=fake, rope_table=fake, frames_written=written,
                            cfg=V.make_config(w))
        return lib.mla_cache_append(ctypes.byref(cache), fake, fake, None, fake, None, first, n,
                                    None)

    sink = synth.workload("sink")                    # W = 7, S = 1: six FIFO frame slots
    assert append(sink, 1, 7, 1) == V.MLA_ERR_RANGE  # frames 1..7: seven FIFO frames
    assert append(sink, 0, 7, 0) != V.MLA_ERR_RANGE  # the sink + six FIFO frames
    assert append(sink, 1, 6, 1) != V.MLA_ERR_RANGE  # exactly W - S FIFO frames
    assert append(sink, 955, 6, 958) != V.MLA_ERR_RANGE
    assert append(sink, 955, 7, 958) == V.MLA_ERR_RANGE
    w4 = synth.workload("tiny", window_frames=4, sink_frames=1)
    assert append(w4, 1, 4, 1) == V.MLA_ERR_RANGE    # frames 1 and 4 would share a slot
    assert append(w4, 1, 3, 1) != V.MLA_ERR_RANGE
    w2 = synth.workload("tiny", window_frames=4, sink_frames=2)
    assert append(w2, 1, 3, 1) != V.MLA_ERR_RANGE    # frame 1 is a sink, 2 and 3 fill the FIFO
    assert append(w2, 1, 4, 1) == V.MLA_ERR_RANGE
    assert append(w2, 0, 4, 0) != V.MLA_ERR_RANGE
    plain = synth.workload("tiny")                   # S = 0: the plain ring, n <= W
    assert append(plain, 0, plain.window_frames, 0) != V.MLA_ERR_RANGE


def _aligned_host(nbytes):
    buf = np.zeros(nbytes + 64, dtype=np.uint8)
    off = (-buf.ctypes.data) % 64
    return buf, ctypes.c_void_p(buf.ctypes.data + off)


def test_host_memory_is_refused():
    """Every buffer must be device memory of the current device (the kernels
    copy tiles with TMA and multicast them within a cluster of this GPU).
    Host buffers are refused before anything is enqueued: MLA_ERR_ARG where a
    GPU is present, MLA_ERR_CUDA here without one (no current device)."""
    lib = V.load()
    w = synth.workload("tiny")
    cfg = V.make_config(w)
    keep, p = [], []
    for nbytes in (w.slots * w.d_c * 2, w.slots * w.d_r * 2, 1024 * w.d_r * 4,
                   64 * 12 * w.d_c * 2, 64 * 12 * w.d_r * 2, 64 * 12, 64 * 12 * w.d_c * 2):
        b, ptr = _aligned_host(nbytes)
        keep.append(b)
        p.append(ptr)
    cache = V.mla_cache(c=p[0], kr=p[1], rope_table=p[2], frames_written=w.window_frames, cfg=cfg)
    rc = lib.mla_attention_forward(ctypes.byref(cache), p[3], p[4], p[5], 64, p[6], None)
    assert rc in (V.MLA_ERR_ARG, V.MLA_ERR_CUDA)
    if rc == V.MLA_ERR_CUDA:
        assert lib.mla_last_cuda_error() != 0
    rc = lib.mla_cache_reset(ctypes.byref(cache), None)
    assert rc in (V.MLA_ERR_ARG, V.MLA_ERR_CUDA)

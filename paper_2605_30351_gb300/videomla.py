"""ctypes binding of libvideomla.so (include/videomla.h), same names as the C ABI.

Argument marshalling only: every step of the cache append and of the
attention runs in the library's CUDA kernels. PyTorch supplies device memory
and streams. There is no fallback: if the library is missing or a call
fails, these functions raise.
"""

import ctypes
import os

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libvideomla.so")

MLA_OK = 0
MLA_ERR_ARG = -1
MLA_ERR_UNSUPPORTED = -2
MLA_ERR_RANGE = -3
MLA_ERR_CUDA = -4
MLA_ERR_TIMEOUT = -5
MLA_ERR_TOO_LARGE = -6
MLA_NOALLOC_SCRATCH_BYTES = 8 * 1024 * 1024

MLA_FLAG_NO_RMSNORM = 1
MLA_FLAG_SIMT = 2
MLA_FLAG_ROTATE_AT_USE = 4

# Every symbol include/videomla.h declares.
EXPORTS = ("mla_rope_table_bytes", "mla_rope_table_fill", "mla_config_check",
           "mla_cache_reset", "mla_cache_append", "mla_attention_forward",
           "mla_absorb_weights", "mla_query_workspace_bytes", "mla_query_prologue",
           "mla_query_prologue_noalloc", "mla_output_projection", "mla_dense_attention_forward",
           "mla_window_workspace_bytes", "mla_attention_window_forward", "mla_decompress_window",
           "mla_selftest_bounded_wait", "mla_status_string", "mla_last_cuda_error", "mla_device_status",
           "mla_debug_rescale_count", "mla_version")


class mla_config(ctypes.Structure):
    _fields_ = [
        ("hidden", ctypes.c_int), ("heads", ctypes.c_int), ("head_dim", ctypes.c_int),
        ("d_c", ctypes.c_int), ("d_r", ctypes.c_int), ("d_q", ctypes.c_int),
        ("rope_pairs_t", ctypes.c_int), ("rope_pairs_h", ctypes.c_int),
        ("rope_pairs_w", ctypes.c_int),
        ("rope_dim_t", ctypes.c_int), ("rope_dim_h", ctypes.c_int), ("rope_dim_w", ctypes.c_int),
        ("rope_theta", ctypes.c_double), ("rope_table_len", ctypes.c_int),
        ("tokens_per_frame", ctypes.c_int), ("window_frames", ctypes.c_int),
        ("batch", ctypes.c_int), ("rms_eps", ctypes.c_float), ("flags", ctypes.c_uint),
        ("sink_frames", ctypes.c_int),
    ]


class mla_cache(ctypes.Structure):
    _fields_ = [
        ("c", ctypes.c_void_p), ("kr", ctypes.c_void_p), ("rope_table", ctypes.c_void_p),
        ("frames_written", ctypes.c_longlong), ("cfg", mla_config),
    ]


class MlaError(RuntimeError):
    def __init__(self, fn, code, lib):
        self.code = code
        msg = lib.mla_status_string(code).decode()
        if code == MLA_ERR_CUDA:
            msg += f" (cudaError {lib.mla_last_cuda_error()})"
        super().__init__(f"{fn} failed: {msg} [{code}]")


_lib = None


def load():
    """Load the in-tree library once; raise if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    P, VP, I, LL = ctypes.POINTER, ctypes.c_void_p, ctypes.c_int, ctypes.c_longlong
    lib.mla_rope_table_bytes.argtypes = [P(mla_config)]
    lib.mla_rope_table_bytes.restype = ctypes.c_ulonglong
    lib.mla_rope_table_fill.argtypes = [P(mla_config), P(ctypes.c_float)]
    lib.mla_config_check.argtypes = [P(mla_config)]
    lib.mla_cache_reset.argtypes = [P(mla_cache), VP]
    lib.mla_cache_append.argtypes = [P(mla_cache), VP, VP, VP, VP, VP, LL, I, VP]
    lib.mla_attention_forward.argtypes = [P(mla_cache), VP, VP, VP, I, VP, VP]
    lib.mla_status_string.argtypes = [I]
    lib.mla_status_string.restype = ctypes.c_char_p
    lib.mla_last_cuda_error.argtypes = []
    lib.mla_device_status.argtypes = [P(I), I]
    lib.mla_debug_rescale_count.argtypes = [P(ctypes.c_ulonglong), I]
    lib.mla_version.argtypes = []
    lib.mla_absorb_weights.argtypes = [P(mla_config), VP, VP, VP, VP, VP, VP, VP, VP, VP]
    lib.mla_query_workspace_bytes.argtypes = [P(mla_config), I]
    lib.mla_query_workspace_bytes.restype = ctypes.c_ulonglong
    lib.mla_query_prologue.argtypes = [P(mla_config), VP, VP, VP, I, VP, ctypes.c_ulonglong, VP,
                                       VP, VP]
    lib.mla_output_projection.argtypes = [P(mla_config), VP, VP, I, VP, VP]
    lib.mla_query_prologue_noalloc.argtypes = [P(mla_config), VP, VP, VP, I, VP, VP, VP]
    lib.mla_dense_attention_forward.argtypes = [P(mla_config), VP, VP, VP, I, I, I, VP, VP]
    lib.mla_decompress_window.argtypes = [P(mla_cache), VP, VP, VP, VP, VP]
    lib.mla_selftest_bounded_wait.argtypes = [ctypes.c_ulonglong, VP]
    lib.mla_window_workspace_bytes.argtypes = [P(mla_config), I]
    lib.mla_window_workspace_bytes.restype = ctypes.c_ulonglong
    lib.mla_attention_window_forward.argtypes = [P(mla_cache), VP, VP, VP, I, VP, VP,
                                                 ctypes.c_ulonglong, VP, VP]
    for name in ("mla_rope_table_fill", "mla_config_check", "mla_cache_reset", "mla_cache_append",
                 "mla_attention_forward", "mla_last_cuda_error", "mla_device_status",
                 "mla_version", "mla_absorb_weights", "mla_query_prologue",
                 "mla_query_prologue_noalloc", "mla_output_projection",
                 "mla_dense_attention_forward", "mla_attention_window_forward",
                 "mla_decompress_window", "mla_selftest_bounded_wait",
                 "mla_debug_rescale_count"):
        getattr(lib, name).restype = I
    _lib = lib
    return lib


def _check(fn, code):
    if code != MLA_OK:
        raise MlaError(fn, code, load())


def make_config(w, flags=0):
    """mla_config from a synth.Workload-like object (a workload with sink
    frames keeps k^R unrotated: the long-rollout window of App. D.4-D.5)."""
    sink = getattr(w, "sink_frames", 0)
    if sink:
        flags |= MLA_FLAG_ROTATE_AT_USE
    return mla_config(
        hidden=w.hidden, heads=w.heads, head_dim=w.head_dim, d_c=w.d_c, d_r=w.d_r, d_q=w.d_q,
        rope_pairs_t=w.rope_pairs[0], rope_pairs_h=w.rope_pairs[1], rope_pairs_w=w.rope_pairs[2],
        rope_dim_t=w.rope_axis_dims[0], rope_dim_h=w.rope_axis_dims[1],
        rope_dim_w=w.rope_axis_dims[2], rope_theta=w.rope_theta,
        rope_table_len=w.rope_table_len, tokens_per_frame=w.tokens_per_frame,
        window_frames=w.window_frames, batch=w.batch, rms_eps=w.rms_eps, flags=flags,
        sink_frames=sink)


def mla_config_check(cfg):
    return load().mla_config_check(ctypes.byref(cfg))


def mla_rope_table_fill(cfg):
    """The RoPE cos/sin table as a float32 NumPy array [L, d_r/2, 2]."""
    lib = load()
    nbytes = lib.mla_rope_table_bytes(ctypes.byref(cfg))
    if nbytes == 0:
        raise MlaError("mla_rope_table_bytes", MLA_ERR_ARG, lib)
    out = np.empty((cfg.rope_table_len, cfg.d_r // 2, 2), dtype=np.float32)
    _check("mla_rope_table_fill",
           lib.mla_rope_table_fill(ctypes.byref(cfg),
                                   out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))))
    return out


def _stream_ptr(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(t, dtype, shape, name):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


class LatentCache:
    """Device buffers of one layer's sliding-window latent cache + the C struct.

    c  bf16 [B, W*T, d_c]; kr bf16 [B, W*T, d_r]; rope fp32 [L, d_r/2, 2].
    """

    def __init__(self, cfg, device="cuda"):
        self.cfg = cfg
        slots = cfg.tokens_per_frame * cfg.window_frames
        self.c = torch.zeros(cfg.batch, slots, cfg.d_c, dtype=torch.bfloat16, device=device)
        self.kr = torch.zeros(cfg.batch, slots, cfg.d_r, dtype=torch.bfloat16, device=device)
        self.rope = torch.from_numpy(mla_rope_table_fill(cfg)).to(device)
        self.struct = mla_cache(c=self.c.data_ptr(), kr=self.kr.data_ptr(),
                                rope_table=self.rope.data_ptr(), frames_written=0, cfg=cfg)

    @property
    def frames_written(self):
        return self.struct.frames_written

    @frames_written.setter
    def frames_written(self, v):
        self.struct.frames_written = int(v)

    @property
    def slots(self):
        return self.cfg.tokens_per_frame * self.cfg.window_frames

    def n_valid(self):
        held = min(self.frames_written, self.cfg.window_frames)
        return held * self.cfg.tokens_per_frame


def mla_cache_reset(cache, stream=None):
    _check("mla_cache_reset",
           load().mla_cache_reset(ctypes.byref(cache.struct), _stream_ptr(stream)))


def mla_cache_append(cache, x, w_dkv, gamma_kv, w_kr, pos, first_frame, n_frames, stream=None):
    cfg = cache.cfg
    n_tok = n_frames * cfg.tokens_per_frame
    bf = torch.bfloat16
    args = (
        _dev(x, bf, (cfg.batch, n_tok, cfg.hidden), "x"),
        _dev(w_dkv, bf, (cfg.d_c, cfg.hidden), "w_dkv"),
        None if gamma_kv is None else _dev(gamma_kv, bf, (cfg.d_c,), "gamma_kv"),
        _dev(w_kr, bf, (cfg.d_r, cfg.hidden), "w_kr"),
        None if pos is None and cfg.flags & MLA_FLAG_ROTATE_AT_USE
        else _dev(pos, torch.int32, (cfg.batch, n_tok, 3), "pos"),
    )
    _check("mla_cache_append",
           load().mla_cache_append(ctypes.byref(cache.struct), *args, int(first_frame),
                                   int(n_frames), _stream_ptr(stream)))


def mla_attention_forward(cache, q_c, q_r, q_pos, o_lat, stream=None):
    cfg = cache.cfg
    Nq = q_c.shape[1]
    bf = torch.bfloat16
    args = (
        _dev(q_c, bf, (cfg.batch, Nq, cfg.heads, cfg.d_c), "q_c"),
        _dev(q_r, bf, (cfg.batch, Nq, cfg.heads, cfg.d_r), "q_r"),
        _dev(q_pos, torch.int32, (cfg.batch, Nq, 3), "q_pos"),
    )
    out = _dev(o_lat, bf, (cfg.batch, Nq, cfg.heads, cfg.d_c), "o_lat")
    _check("mla_attention_forward",
           load().mla_attention_forward(ctypes.byref(cache.struct), *args, int(Nq), out,
                                        _stream_ptr(stream)))


def mla_window_workspace_bytes(cfg, Nq):
    return int(load().mla_window_workspace_bytes(ctypes.byref(cfg), int(Nq)))


def mla_attention_window_forward(cache, q_c, q_r, q_pos, frame_hw, workspace, o_lat, stream=None):
    """Attention over the assembled sink + FIFO window with window-relative
    RoPE (App. D.4, D.5); q_pos holds absolute frames, frame_hw [T, 2] the
    (h, w) of every token of a latent frame."""
    cfg = cache.cfg
    Nq = q_c.shape[1]
    bf = torch.bfloat16
    if not (isinstance(workspace, torch.Tensor) and workspace.is_cuda and workspace.is_contiguous()):
        raise TypeError("workspace must be a contiguous CUDA tensor")
    _check("mla_attention_window_forward",
           load().mla_attention_window_forward(
               ctypes.byref(cache.struct),
               _dev(q_c, bf, (cfg.batch, Nq, cfg.heads, cfg.d_c), "q_c"),
               _dev(q_r, bf, (cfg.batch, Nq, cfg.heads, cfg.d_r), "q_r"),
               _dev(q_pos, torch.int32, (cfg.batch, Nq, 3), "q_pos"), int(Nq),
               _dev(frame_hw, torch.int32, (cfg.tokens_per_frame, 2), "frame_hw"),
               ctypes.c_void_p(workspace.data_ptr()),
               workspace.numel() * workspace.element_size(),
               _dev(o_lat, bf, (cfg.batch, Nq, cfg.heads, cfg.d_c), "o_lat"),
               _stream_ptr(stream)))


def mla_decompress_window(cache, w_uk, w_uv, k, v, stream=None):
    """Expand the latent cache into per-head keys [W_up^K c | k] and values
    W_up^V c, both [B, H, W*T, head_dim] (the decompress-then-dense form)."""
    cfg = cache.cfg
    H, dh, dr, dc = cfg.heads, cfg.head_dim, cfg.d_r, cfg.d_c
    shape = (cfg.batch, H, cache.slots, dh)
    bf = torch.bfloat16
    _check("mla_decompress_window",
           load().mla_decompress_window(
               ctypes.byref(cache.struct), _dev(w_uk, bf, (H, dh - dr, dc), "w_uk"),
               _dev(w_uv, bf, (H, dh, dc), "w_uv"), _dev(k, bf, shape, "k"),
               _dev(v, bf, shape, "v"), _stream_ptr(stream)))


def absorbed_weight_shapes(cfg):
    """Shapes of (w_qcat, w_b) that mla_absorb_weights writes."""
    return ((cfg.heads * (cfg.d_c + cfg.d_r), cfg.d_q), (cfg.hidden, cfg.heads * cfg.d_c))


def mla_absorb_weights(cfg, w_uq, w_uk, w_qr, gamma_q, w_uv, w_o, stream=None):
    """Absorbed query and output weights (App. E) as new bf16 CUDA tensors."""
    H, dc, dr, dq, d, dh = cfg.heads, cfg.d_c, cfg.d_r, cfg.d_q, cfg.hidden, cfg.head_dim
    dn = dh - dr
    bf = torch.bfloat16
    args = (
        _dev(w_uq, bf, (H, dn, dq), "w_uq"), _dev(w_uk, bf, (H, dn, dc), "w_uk"),
        _dev(w_qr, bf, (H, dr, dq), "w_qr"),
        None if gamma_q is None else _dev(gamma_q, bf, (dq,), "gamma_q"),
        _dev(w_uv, bf, (H, dh, dc), "w_uv"), _dev(w_o, bf, (d, H * dh), "w_o"),
    )
    sq, sb = absorbed_weight_shapes(cfg)
    w_qcat = torch.empty(sq, dtype=bf, device=w_uq.device)
    w_b = torch.empty(sb, dtype=bf, device=w_uq.device)
    _check("mla_absorb_weights",
           load().mla_absorb_weights(ctypes.byref(cfg), *args, ctypes.c_void_p(w_qcat.data_ptr()),
                                     ctypes.c_void_p(w_b.data_ptr()), _stream_ptr(stream)))
    return w_qcat, w_b


def mla_query_workspace_bytes(cfg, Nq):
    return int(load().mla_query_workspace_bytes(ctypes.byref(cfg), int(Nq)))


def mla_query_prologue(cfg, x, w_dq, w_qcat, workspace, q_c, q_r, stream=None):
    Nq = x.shape[1]
    bf = torch.bfloat16
    H, dc, dr, dq, d = cfg.heads, cfg.d_c, cfg.d_r, cfg.d_q, cfg.hidden
    if not (isinstance(workspace, torch.Tensor) and workspace.is_cuda and workspace.is_contiguous()):
        raise TypeError("workspace must be a contiguous CUDA tensor")
    _check("mla_query_prologue",
           load().mla_query_prologue(
               ctypes.byref(cfg), _dev(x, bf, (cfg.batch, Nq, d), "x"),
               _dev(w_dq, bf, (dq, d), "w_dq"), _dev(w_qcat, bf, (H * (dc + dr), dq), "w_qcat"),
               int(Nq), ctypes.c_void_p(workspace.data_ptr()),
               workspace.numel() * workspace.element_size(),
               _dev(q_c, bf, (cfg.batch, Nq, H, dc), "q_c"),
               _dev(q_r, bf, (cfg.batch, Nq, H, dr), "q_r"), _stream_ptr(stream)))


def mla_query_prologue_noalloc(cfg, x, w_dq, w_qcat, q_c, q_r, stream=None):
    """The query prologue for callers that cannot allocate device memory: the
    intermediate buffer is the library's fixed scratch (see the C header for
    its size limit and the rule that overlapping calls race on it)."""
    Nq = x.shape[1]
    bf = torch.bfloat16
    H, dc, dr, dq, d = cfg.heads, cfg.d_c, cfg.d_r, cfg.d_q, cfg.hidden
    _check("mla_query_prologue_noalloc",
           load().mla_query_prologue_noalloc(
               ctypes.byref(cfg), _dev(x, bf, (cfg.batch, Nq, d), "x"),
               _dev(w_dq, bf, (dq, d), "w_dq"), _dev(w_qcat, bf, (H * (dc + dr), dq), "w_qcat"),
               int(Nq), _dev(q_c, bf, (cfg.batch, Nq, H, dc), "q_c"),
               _dev(q_r, bf, (cfg.batch, Nq, H, dr), "q_r"), _stream_ptr(stream)))


def mla_output_projection(cfg, o_lat, w_b, y, stream=None):
    Nq = o_lat.shape[1]
    bf = torch.bfloat16
    _check("mla_output_projection",
           load().mla_output_projection(
               ctypes.byref(cfg), _dev(o_lat, bf, (cfg.batch, Nq, cfg.heads, cfg.d_c), "o_lat"),
               _dev(w_b, bf, (cfg.hidden, cfg.heads * cfg.d_c), "w_b"), int(Nq),
               _dev(y, bf, (cfg.batch, Nq, cfg.hidden), "y"), _stream_ptr(stream)))


def mla_dense_attention_forward(cfg, q, k, v, n_valid, o, stream=None):
    """Dense per-head baseline: q [B, Nq, H, d_h], k/v [B, H, slots, d_h]."""
    B, Nq, H, dh = cfg.batch, q.shape[1], cfg.heads, cfg.head_dim
    slots = k.shape[2]
    bf = torch.bfloat16
    _check("mla_dense_attention_forward",
           load().mla_dense_attention_forward(
               ctypes.byref(cfg), _dev(q, bf, (B, Nq, H, dh), "q"),
               _dev(k, bf, (B, H, slots, dh), "k"), _dev(v, bf, (B, H, slots, dh), "v"),
               int(slots), int(n_valid), int(Nq), _dev(o, bf, (B, Nq, H, dh), "o"),
               _stream_ptr(stream)))


def mla_selftest_bounded_wait(limit_ns, stream=None):
    """Make one bounded device wait run out (nothing arrives on its barrier)."""
    _check("mla_selftest_bounded_wait",
           load().mla_selftest_bounded_wait(int(limit_ns), _stream_ptr(stream)))


def mla_device_status(clear=True):
    st = ctypes.c_int(0)
    _check("mla_device_status", load().mla_device_status(ctypes.byref(st), int(bool(clear))))
    return st.value


def mla_debug_rescale_count(clear=True):
    """Rows whose online softmax rescaled its output (debug build only; a
    release build raises MlaError with MLA_ERR_UNSUPPORTED)."""
    n = ctypes.c_ulonglong(0)
    _check("mla_debug_rescale_count",
           load().mla_debug_rescale_count(ctypes.byref(n), int(bool(clear))))
    return n.value

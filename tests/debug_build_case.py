"""Helper run in a subprocess by test_gpu_debug_build.py: loads the library
named on the command line (release or debug build), runs a fixed set of
calls (append + attention on the 21-frame ring, the sink window, the
decompression, the query prologue and output projection; the append's
cluster and split forms and the split-output attention at d_c = 256 and 512;
the layer GEMMs' paired-SM form at four chunks; the online softmax's
rescale branch in the absorbed and dense kernels) on
seeded inputs and saves every output, the device status word and the debug
build's count of softmax rescales (-1 for the release build, which does not
count)."""

import os
import sys

import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

from paper_2605_30351_gb300 import synth  # noqa: E402
from paper_2605_30351_gb300 import videomla as V  # noqa: E402


def main(lib_path, out_path):
    V.LIB_PATH = lib_path
    V._lib = None
    V.load()
    V.mla_device_status(clear=True)
    out = {}
    for sink in (0, 1):
        w = synth.workload("tiny", grid_h=10, grid_w=10, window_frames=4, sink_frames=sink, batch=2)
        wt = {k: t.cuda() for k, t in synth.draw_layer_weights(w, 31).items()}
        cfg = V.make_config(w)
        cache = V.LatentCache(cfg)
        V.mla_cache_reset(cache)
        T = w.tokens_per_frame
        for f in range(7):
            x = synth.draw_tokens(w, T, 40 + f).cuda()
            pos = None if sink else synth.grid_positions(w, f, 1).cuda()
            V.mla_cache_append(cache, x, wt["w_dkv"], wt["gamma_kv"], wt["w_kr"], pos, f, 1)
        q_c, q_r = synth.draw_queries(w, T, 50)
        q_pos = synth.grid_positions(w, 6, 1).cuda()
        o = torch.empty(w.batch, T, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
        if sink:
            ws = torch.empty(V.mla_window_workspace_bytes(cfg, T), dtype=torch.uint8, device="cuda")
            V.mla_attention_window_forward(cache, q_c.cuda(), q_r.cuda(), q_pos,
                                           synth.frame_coords(w).cuda(), ws, o)
        else:
            V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), q_pos, o)
            k = torch.empty(w.batch, w.heads, w.slots, w.head_dim, dtype=torch.bfloat16,
                            device="cuda")
            v = torch.empty_like(k)
            V.mla_decompress_window(cache, wt["w_uk"], wt["w_uv"], k, v)
            out["k"], out["v"] = k.cpu(), v.cpu()
            w_qcat, w_b = V.mla_absorb_weights(cfg, wt["w_uq"], wt["w_uk"], wt["w_qr"],
                                               wt["gamma_q"], wt["w_uv"], wt["w_o"])
            x = synth.draw_tokens(w, T, 60).cuda()
            wsq = torch.empty(V.mla_query_workspace_bytes(cfg, T), dtype=torch.uint8, device="cuda")
            qc2 = torch.empty(w.batch, T, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
            qr2 = torch.empty(w.batch, T, w.heads, w.d_r, dtype=torch.bfloat16, device="cuda")
            V.mla_query_prologue(cfg, x, wt["w_dq"], w_qcat, wsq, qc2, qr2)
            y = torch.empty(w.batch, T, w.hidden, dtype=torch.bfloat16, device="cuda")
            V.mla_output_projection(cfg, o, w_b, y)
            out["q_c"], out["q_r"], out["y"] = qc2.cpu(), qr2.cpu(), y.cpu()
        torch.cuda.synchronize()
        out[f"c{sink}"], out[f"kr{sink}"], out[f"o{sink}"] = cache.c.cpu(), cache.kr.cpu(), o.cpu()
    # the other launch forms: a cluster of 4 CTAs per token tile (d_c = 256) and
    # the split append and split-output attention of d_c = 512
    for d_c in (256, 512):
        w = synth.workload("tiny", grid_h=10, grid_w=10, window_frames=3, batch=2, d_c=d_c,
                           rope_pairs=(6, 5, 5))
        wt = {k: t.cuda() for k, t in synth.draw_layer_weights(w, 33).items()}
        cache = V.LatentCache(V.make_config(w))
        V.mla_cache_reset(cache)
        T = w.tokens_per_frame
        for f in range(4):
            x = synth.draw_tokens(w, T, 70 + f).cuda()
            V.mla_cache_append(cache, x, wt["w_dkv"], wt["gamma_kv"], wt["w_kr"],
                               synth.grid_positions(w, f, 1).cuda(), f, 1)
        q_c, q_r = synth.draw_queries(w, T, 80)
        o = torch.empty(w.batch, T, w.heads, d_c, dtype=torch.bfloat16, device="cuda")
        V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(), synth.grid_positions(w, 3, 1).cuda(),
                                o)
        torch.cuda.synchronize()
        out[f"c_{d_c}"], out[f"kr_{d_c}"], out[f"o_{d_c}"] = cache.c.cpu(), cache.kr.cpu(), o.cpu()
    # the layer GEMMs in their paired-SM form (four Wan chunks: 147 row tiles,
    # the last pair half past the tokens)
    w = synth.workload("wan", batch=4)
    cfg = V.make_config(w)
    wt = {k: t.cuda() for k, t in synth.draw_layer_weights(w, 37).items()}
    w_qcat, w_b = V.mla_absorb_weights(cfg, wt["w_uq"], wt["w_uk"], wt["w_qr"], wt["gamma_q"],
                                       wt["w_uv"], wt["w_o"])
    nq = w.chunk_tokens
    x = synth.draw_tokens(w, nq, 87).cuda()
    wsq = torch.empty(V.mla_query_workspace_bytes(cfg, nq), dtype=torch.uint8, device="cuda")
    qc4 = torch.empty(4, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    qr4 = torch.empty(4, nq, w.heads, w.d_r, dtype=torch.bfloat16, device="cuda")
    V.mla_query_prologue(cfg, x, wt["w_dq"], w_qcat, wsq, qc4, qr4)
    y4 = torch.empty(4, nq, w.hidden, dtype=torch.bfloat16, device="cuda")
    V.mla_output_projection(cfg, qc4, w_b, y4)
    torch.cuda.synchronize()
    out["q_c4"], out["q_r4"], out["y4"] = qc4.cpu(), qr4.cpu(), y4.cpu()
    # the online softmax's rescale branch: a dominant key in the last key
    # block for a third of the rows, absorbed (390 keys) and dense (500 keys)
    from test_gpu_softmax import absorbed_inputs, dense_inputs
    try:
        V.mla_debug_rescale_count(clear=True)
    except V.MlaError as e:
        assert e.code == V.MLA_ERR_UNSUPPORTED  # the release build does not count
    w = synth.workload("tiny", grid_h=10, grid_w=13, window_frames=3, batch=2,
                       rope_pairs=(6, 5, 5))
    q_c, q_r, c, k, _ = absorbed_inputs(w, 40, "late", 90)
    cache = V.LatentCache(V.make_config(w))
    cache.c.copy_(c)
    cache.kr.copy_(k)
    cache.frames_written = w.window_frames
    o = torch.empty(w.batch, 40, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
    V.mla_attention_forward(cache, q_c.cuda(), q_r.cuda(),
                            synth.grid_positions(w, 2, 1)[:, :40].contiguous().cuda(), o)
    wd = synth.workload("tiny", batch=2)
    q, kd, vd, _ = dense_inputs(wd, 300, 500, "late", 91)
    od = torch.empty(q.shape, dtype=torch.bfloat16, device="cuda")
    V.mla_dense_attention_forward(V.make_config(wd), q.cuda(), kd.cuda(), vd.cuda(), 500, od)
    torch.cuda.synchronize()
    out["o_late"], out["o_dense_late"] = o.cpu(), od.cpu()
    try:
        out["rescales"] = V.mla_debug_rescale_count(clear=True)
    except V.MlaError as e:
        assert e.code == V.MLA_ERR_UNSUPPORTED
        out["rescales"] = -1
    out["status"] = V.mla_device_status(clear=True)
    torch.save(out, out_path)


if __name__ == "__main__":
    main(sys.argv[1], sys.argv[2])

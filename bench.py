"""Benchmark of one VideoMLA layer-chunk on GB300: cache append + absorbed MLA
attention at the Wan2.1-1.3B shape (4680-query chunk, 32760-key window,
12 heads, d_c = 192, d_r = 32, batch 1), through the C ABI.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload wan|wan30|rollout|sink]
                  [--sweep dc|memcap|layer|crossover]

One step = mla_cache_append of the current 3-frame chunk + mla_attention_forward
of that chunk against the full 21-frame window (one layer, one denoising step;
30 layers for wan30; batch 4 for rollout and sink, sink using the 1 + 6 frame
window with rotate-at-use RoPE). Prints one JSON line. The --sweep modes print
one JSON line each: the latent-size sweep next to the dense baseline, the
memory-cap batch sweep, the whole layer by phase, and absorbed vs
decompress-then-dense by query-chunk size.

Single GPU only. The attention kernels share key tiles among the CTAs of a
cluster by TMA multicast within this GPU's memory, which may only run in
single-GPU jobs; under torchrun with more than one rank the GPU arm prints an
"unavailable" line (rank 0) and every rank exits 0. The reference arm (the
float64 oracle on the host cores) runs on rank 0 alone.
"""

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2605_30351_gb300 import synth  # noqa: E402

METRIC = "MLA attention TFLOP/s & % bf16 peak; ms per chunk per layer at Wan-1.3B shape"
UNIT = "TFLOP/s"
N_SETS = 4  # rotating input sets: 4 x 76 MB > 129 MB L2, so no set is L2-resident
PROFILES = os.path.join(ROOT, "profiles")


def workload_desc(w):
    layers = f"{w.layers} layers (distinct weights and caches), " if w.layers > 1 else ""
    pos = f"; latent frames up to {w.last_frame - 1} (ring wrapped)" if w.last_frame > w.window_frames else ""
    frames = (f"{w.window_frames} frames: {w.sink_frames} sink + {w.window_frames - w.sink_frames}"
              f" newest, k^R rotated at use at window-relative positions" if w.sink_frames
              else f"{w.window_frames} frames")
    return (f"Wan2.1-1.3B attention layer: {w.chunk_tokens}-query chunk "
            f"({w.chunk_frames} latent frames of {w.grid_h}x{w.grid_w}) x {w.slots}-key window "
            f"({frames}), {w.heads} heads, d_c={w.d_c}, d_r={w.d_r}, "
            f"batch {w.batch}; step = {layers}cache append + attention{pos}")


def flops_per_layer(w):
    rows = w.batch * w.chunk_tokens * w.heads
    attn = 2.0 * rows * w.slots * (w.d_c + w.d_r) + 2.0 * rows * w.slots * w.d_c
    append = 2.0 * w.batch * w.chunk_tokens * w.hidden * (w.d_c + w.d_r)
    return attn, append


def append_bytes(w):
    """Algorithmic HBM bytes of one append (one layer): x, both weights, gamma,
    positions in; c and k rows out."""
    n = w.batch * w.chunk_tokens
    return (n * w.hidden * 2 + (w.d_c + w.d_r) * w.hidden * 2 + w.d_c * 2 + n * 3 * 4
            + n * (w.d_c + w.d_r) * 2)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


def kernel_source_hash(name):
    src = os.path.join(ROOT, "paper_2605_30351_gb300", "csrc", name)
    with open(src, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def append_kernel_name(w):
    """The append kernel the library launches for this shape: a cluster of
    d_c/64 CTAs per token tile when those CTAs fit in one wave (the launch
    also checks that the clusters are co-resident), else one CTA per tile."""
    tiles = -(-w.chunk_tokens // 128)
    sms = torch.cuda.get_device_properties(0).multi_processor_count if torch.cuda.is_available() else 152
    if 128 <= w.d_c <= 256 and tiles * w.batch * (w.d_c // 64) <= sms:
        return f"mla_append_tc_cluster_kernel<{w.d_c},{w.d_r}>"
    return f"mla_append_tc_kernel<{w.d_c},{w.d_r}>"


def profiled_traffic(summary, kernel_src):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current kernel source (else None)."""
    p = os.path.join(PROFILES, summary)
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    if d.get("kernel_source_sha256_16") != kernel_source_hash(kernel_src):
        return None
    return d.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [ln for ln in out.splitlines() if ln.strip()]

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in getattr(self, "lines", []):
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for name, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        loaded = [s for s in sm if s > 0.5 * (mx or max(sm))] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------- CPU oracle
# The float64 oracle, as it stands, timed on every host core: one spawned
# worker process per core (spawn, so no worker inherits a CUDA context), each
# running the oracle single-threaded on its own slice of query tokens. Both
# the GPU arm's cpu_baseline leg and the reference arm time the SAME sample:
# query tokens 0 .. P*TOKENS_PER_WORKER-1 of the chunk (P = worker count),
# each with its cache append and its 12 heads' attention against the full
# window.
TOKENS_PER_WORKER = 1
_ORACLE = None  # per-worker state (inputs drawn from the same seeds in every worker)


def _oracle_state(w, seed):
    from oracle import mla_oracle as O

    spec = O.RopeSpec(w.rope_pairs, w.rope_axis_dims, w.rope_theta)
    weights = synth.draw_layer_weights(w, seed)
    f64 = lambda t: t.float().numpy().astype(np.float64)
    st = {"w": w, "spec": spec, "wd": f64(weights["w_dkv"]), "wk": f64(weights["w_kr"]),
          "g": f64(weights["gamma_kv"])}
    c, k = synth.draw_cache_rows(w, w.slots, seed + 1, batch=1)
    st["c"], st["k"] = f64(c[0]), f64(k[0])
    st["win"] = None
    if w.sink_frames:
        # the window oracle: a cache holding the sink frame and the newest
        # frames with k^R unrotated, rotated at window-local times per call
        win = O.OracleCache(1, w.tokens_per_frame, w.window_frames, w.d_c, w.d_r,
                            sink_frames=w.sink_frames)
        T = w.tokens_per_frame
        first_local = w.last_frame - (w.window_frames - w.sink_frames)
        for f in list(range(w.sink_frames)) + list(range(first_local, w.last_frame)):
            s0 = O.sink_ring_slot(f, 0, T, w.window_frames, w.sink_frames)
            win.frame_of_slot[s0:s0 + T] = f
            win.pos_of_slot[0, s0:s0 + T] = synth.grid_positions(w, f, 1, batch=1)[0].numpy()
        win.c[0], win.kr[0] = st["c"], st["k"]
        win.frames_written = w.last_frame
        st["win"] = win
    q_c, q_r = synth.draw_queries(w, w.chunk_tokens, seed + 2, batch=1)
    x = synth.draw_tokens(w, w.chunk_tokens, seed + 3, batch=1)
    pos = synth.grid_positions(w, (w.last_frame if w.sink_frames else w.window_frames)
                               - w.chunk_frames, w.chunk_frames, batch=1)
    st["q_c"], st["q_r"], st["x"], st["pos"] = f64(q_c[0]), f64(q_r[0]), f64(x), pos.numpy()
    return st


def _oracle_init(w, seed):
    global _ORACLE
    _ORACLE = _oracle_state(w, seed)


def _oracle_ready(_):
    return _ORACLE is not None


def _oracle_slice(start, stop):
    """Append + attention of query tokens [start, stop) with the oracle; returns
    (flops, cpu seconds of this process)."""
    from oracle import mla_oracle as O

    st = _ORACLE
    w, spec = st["w"], st["spec"]
    sl = slice(start, stop)
    n = stop - start
    t0 = time.process_time()
    oc = O.OracleCache(1, w.tokens_per_frame, w.window_frames, w.d_c, w.d_r)
    oc.T = n  # one partial "frame" of n tokens: the same arithmetic per token
    O.cache_append(oc, st["x"][:, sl], st["wd"], st["wk"], st["pos"][:, sl], 0, 1, gamma=st["g"],
                   eps=w.rms_eps, spec=None if w.sink_frames else spec)
    if w.sink_frames:
        O.window_attention(st["win"], 0, st["q_c"][sl], st["q_r"][sl], st["pos"][0, sl],
                           w.head_dim, spec)
    else:
        O.latent_attention(st["q_c"][sl], st["q_r"][sl], st["pos"][0, sl], st["c"], st["k"],
                           w.head_dim, spec)
    fl = 2.0 * n * w.hidden * (w.d_c + w.d_r) + O.latent_attention_flops(
        n * w.heads, w.slots, w.d_c, w.d_r)
    return fl, time.process_time() - t0


class OraclePool:
    """One spawned single-threaded oracle worker per host core: `cores` in the
    JSON line is that worker count (one thread each); cpu_utilisation is the
    workers' CPU time over the wall time of the rounds, per worker."""

    def __init__(self, w, seed=5):
        import multiprocessing as mp

        self.w = w
        self.procs = len(os.sched_getaffinity(0))
        self.tokens = min(w.chunk_tokens, self.procs * TOKENS_PER_WORKER)
        saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS",
                                                "MKL_NUM_THREADS")}
        for k in saved:
            os.environ[k] = "1"  # one thread per worker: the pool supplies the parallelism
        try:
            self.pool = mp.get_context("spawn").Pool(self.procs, initializer=_oracle_init,
                                                     initargs=(w, seed))
        finally:
            for k, v in saved.items():
                if v is None:
                    os.environ.pop(k, None)
                else:
                    os.environ[k] = v
        assert all(self.pool.map(_oracle_ready, range(self.procs), chunksize=1))

    def round(self):
        """The whole sample once: (flops, wall seconds, cpu seconds)."""
        slices = [(a, min(a + TOKENS_PER_WORKER, self.tokens))
                  for a in range(0, self.tokens, TOKENS_PER_WORKER)]
        t0 = time.perf_counter()
        res = self.pool.starmap(_oracle_slice, slices, chunksize=1)
        wall = time.perf_counter() - t0
        return sum(r[0] for r in res), wall, sum(r[1] for r in res)

    def describe(self, wall, rounds):
        w = self.w
        return (f"float64 NumPy oracle, {self.procs} single-threaded worker processes: append + "
                f"attention of query tokens 0..{self.tokens - 1} of the {w.chunk_tokens}-token "
                f"chunk (x{w.heads} heads, {TOKENS_PER_WORKER} per worker) against the "
                f"full {w.slots}-key window; {rounds} round(s), {wall:.1f} s")

    def close(self):
        self.pool.terminate()
        self.pool.join()


def cpu_oracle_sample(w, budget_s=12.0, pool=None):
    """Time the oracle on the fixed sample, repeated for about budget_s."""
    own = pool is None
    pool = pool or OraclePool(w)
    try:
        fl = wall = cpu = 0.0
        rounds = 0
        while rounds == 0 or wall < budget_s:
            f, t, c = pool.round()
            fl, wall, cpu, rounds = fl + f, wall + t, cpu + c, rounds + 1
        return {
            "value": fl / wall / 1e12,
            "unit": UNIT,
            "cores": pool.procs,
            "cpu_utilisation": cpu / wall / pool.procs,
            "host_cores_available": len(os.sched_getaffinity(0)),
            "kind": "oracle",
            "sample": pool.describe(wall, rounds),
            "seconds": wall,
        }
    finally:
        if own:
            pool.close()


# ------------------------------------------------------------------ GPU arm
class LayerSet:
    """One layer's device state: weights, a full cache, the step's inputs."""

    def __init__(self, w, seed, V):
        self.w = w
        wt = synth.draw_layer_weights(w, seed)
        self.w_dkv = wt["w_dkv"].cuda()
        self.w_kr = wt["w_kr"].cuda()
        self.gamma = wt["gamma_kv"].cuda()
        self.cache = V.LatentCache(V.make_config(w))
        c, k = synth.draw_cache_rows(w, w.slots, seed + 1)
        self.cache.c.copy_(c)
        self.cache.kr.copy_(k)
        self.cache.frames_written = w.last_frame
        self.first = w.last_frame - w.chunk_frames
        self.x = synth.draw_tokens(w, w.chunk_tokens, seed + 2).cuda()
        self.pos = synth.grid_positions(w, self.first, w.chunk_frames).cuda()
        q_c, q_r = synth.draw_queries(w, w.chunk_tokens, seed + 3)
        self.q_c, self.q_r = q_c.cuda(), q_r.cuda()
        self.o = torch.empty(w.batch, w.chunk_tokens, w.heads, w.d_c, dtype=torch.bfloat16,
                             device="cuda")
        # long-rollout window (sink frames, k^R unrotated): assembled per call
        self.window = w.sink_frames > 0
        if self.window:
            self.hw = synth.frame_coords(w).cuda()
            self.ws = torch.empty(V.mla_window_workspace_bytes(self.cache.cfg, w.chunk_tokens),
                                  dtype=torch.uint8, device="cuda")


def run_ours(args, w):
    from paper_2605_30351_gb300 import videomla as V

    # the oracle's worker processes start before the first GPU call (spawned,
    # so none of them holds a CUDA context); they are timed after the GPU run
    pool = None if args.no_cpu_baseline else OraclePool(w)
    torch.cuda.set_device(0)
    V.load()
    stream = torch.cuda.current_stream()
    # one set per layer of a step, or N_SETS rotating sets for a one-layer step
    n_sets = max(w.layers, N_SETS)
    sets = [LayerSet(w, 1000 + 17 * i, V) for i in range(n_sets)]
    attn_l, app_l = flops_per_layer(w)
    attn_fl, app_fl = attn_l * w.layers, app_l * w.layers

    def layer(s, ev=None):
        if ev is not None:
            ev[0].record(stream)
        V.mla_cache_append(s.cache, s.x, s.w_dkv, s.gamma, s.w_kr, None if s.window else s.pos,
                           s.first, w.chunk_frames, stream)
        if ev is not None:
            ev[1].record(stream)
        if s.window:
            V.mla_attention_window_forward(s.cache, s.q_c, s.q_r, s.pos, s.hw, s.ws, s.o, stream)
        else:
            V.mla_attention_forward(s.cache, s.q_c, s.q_r, s.pos, s.o, stream)
        if ev is not None:
            ev[2].record(stream)

    def step(i, evs=None):
        for L in range(w.layers):
            layer(sets[(i * w.layers + L) % n_sets], None if evs is None else evs[L])

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    assert V.mla_device_status(clear=True) == V.MLA_OK

    # The timed region: K steps back to back between two events (an event
    # between kernels makes the GPU finish one before the next is set up, so
    # the per-kernel events go in a second pass below). Clocks are sampled
    # over both passes.
    ev = [[tuple(torch.cuda.Event(enable_timing=True) for _ in range(3))
           for _ in range(w.layers)] for _ in range(args.steps)]
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    with ClockSampler(0) as clk:
        t_start.record(stream)
        for i in range(args.steps):
            step(i)
        t_end.record(stream)
        torch.cuda.synchronize()
        # kernel durations: the same K steps with events around every launch
        for i in range(args.steps):
            step(i, ev[i])
        torch.cuda.synchronize()
        # the steps' appends alone, back to back between two events: the
        # append's duration without an event on either side of each launch
        # (which costs a short kernel like this one several microseconds)
        b0 = torch.cuda.Event(enable_timing=True)
        b1 = torch.cuda.Event(enable_timing=True)
        b0.record(stream)
        for i in range(args.steps):
            for L in range(w.layers):
                s = sets[(i * w.layers + L) % n_sets]
                V.mla_cache_append(s.cache, s.x, s.w_dkv, s.gamma, s.w_kr,
                                   None if s.window else s.pos, s.first, w.chunk_frames, stream)
        b1.record(stream)
        torch.cuda.synchronize()
    ms_total = t_start.elapsed_time(t_end)
    app_b2b_ms = b0.elapsed_time(b1) / (args.steps * w.layers)
    app_ms_l = [e[0].elapsed_time(e[1]) for es in ev for e in es]
    attn_ms = [e[1].elapsed_time(e[2]) for es in ev for e in es]
    ms_max = ms_total
    status = V.mla_device_status(clear=True)
    if status != V.MLA_OK:
        raise RuntimeError(f"device status {status} after the timed region")

    # end to end through the public API with pinned host buffers: H2D of the
    # step's inputs, append + attention, D2H of the latent output
    h_sets = []
    n_e2e = max(2, w.layers)
    for s in sets[:n_e2e]:
        h_sets.append({"x": s.x.cpu().pin_memory(), "q_c": s.q_c.cpu().pin_memory(),
                       "q_r": s.q_r.cpu().pin_memory(), "pos": s.pos.cpu().pin_memory(),
                       "o": torch.empty_like(s.o, device="cpu").pin_memory()})
    h2d = w.layers * sum(h_sets[0][k].numel() * h_sets[0][k].element_size()
                         for k in ("x", "q_c", "q_r", "pos"))
    d2h = w.layers * h_sets[0]["o"].numel() * h_sets[0]["o"].element_size()
    e2e_steps = max(3, args.steps // 4)
    if w.layers > 1:
        e2e_steps = max(3, min(e2e_steps, 10))

    # Pipelined: each (step, layer) unit has its own device set; its inputs
    # go up on one copy stream and its output comes back on another, so the
    # copies of neighbouring units overlap the kernels of this one.
    h2d_stream, d2h_stream = torch.cuda.Stream(), torch.cuda.Stream()
    uploaded = [torch.cuda.Event() for _ in range(n_e2e)]
    computed = [torch.cuda.Event() for _ in range(n_e2e)]
    downloaded = [torch.cuda.Event() for _ in range(n_e2e)]
    used = [False] * n_e2e

    def upload(u):
        j = u % n_e2e
        s, h = sets[j], h_sets[j]
        with torch.cuda.stream(h2d_stream):
            if used[j]:
                h2d_stream.wait_event(computed[j])  # the set's inputs were last read there
            s.x.copy_(h["x"], non_blocking=True)
            s.q_c.copy_(h["q_c"], non_blocking=True)
            s.q_r.copy_(h["q_r"], non_blocking=True)
            s.pos.copy_(h["pos"], non_blocking=True)
            uploaded[j].record(h2d_stream)

    def compute_and_d2h(u):
        j = u % n_e2e
        s, h = sets[j], h_sets[j]
        stream.wait_event(uploaded[j])
        if used[j]:
            stream.wait_event(downloaded[j])  # the set's output buffer is free again
        layer(s)
        computed[j].record(stream)
        used[j] = True
        with torch.cuda.stream(d2h_stream):
            d2h_stream.wait_event(computed[j])
            h["o"].copy_(s.o, non_blocking=True)
            downloaded[j].record(d2h_stream)

    def e2e_run(n_steps):
        units = n_steps * w.layers
        upload(0)
        for u in range(units):
            if u + 1 < units:
                upload(u + 1)
            compute_and_d2h(u)
        stream.wait_stream(d2h_stream)

    e2e_run(2)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    h2d_stream.wait_event(e0)
    e2e_run(e2e_steps)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)

    # the append alone at batch 4 (a rollout batch), where the HBM bar applies
    append_b4 = time_append_b4(w, V, stream) if w.batch == 1 and w.layers == 1 else None

    peaks = load_peaks()
    ms_step = ms_max / args.steps
    attn_ms_mean = statistics.fmean(attn_ms)
    achieved = attn_l / (attn_ms_mean * 1e-3) / 1e12
    app_ms = statistics.fmean(app_ms_l)
    # the burst peak for a kernel timed over a short region, the sustained one
    # (a seconds-long loop under the power cap) once the timed region is that long
    if ms_max >= 1000.0:
        peak, peak_kind = peaks["bf16_tflops_sustained"], "sustained"
        peak_why = f"timed region {ms_max / 1e3:.1f} s"
    else:
        peak, peak_kind = peaks["bf16_tflops"], "burst"
        peak_why = f"timed region {ms_max:.0f} ms"
    out = {
        "metric": METRIC,
        "value": tflops(attn_fl + app_fl, ms_step),
        "unit": UNIT,
        "n_gpus": 1,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded Gaussian activations, weights N(0,1/fan_in), "
                "cache rows N(0,1)); no dataset or trained weights",
        "config": {
            "workload": workload_desc(w),
            "queries": w.chunk_tokens * w.heads, "keys": w.slots, "heads": w.heads,
            "d_c": w.d_c, "d_r": w.d_r, "hidden": w.hidden, "batch": w.batch,
            "rope_pairs_thw": list(w.rope_pairs),
            "l2": f"inputs larger than L2: {N_SETS} rotating layer sets "
                  f"(~{N_SETS * 76} MB), one per step",
            "parallelism": "single GPU",
        },
        "ms_per_layer": ms_step / w.layers,
        "attention_ms": attn_ms_mean,
        "append_ms": app_ms,
        "roofline": {
            "bound": "tensor", "achieved": achieved, "peak": peak,
            "unit": "TFLOP/s", "frac": achieved / peak,
            "frac_of_burst": achieved / peaks["bf16_tflops"],
            "frac_of_sustained": achieved / peaks["bf16_tflops_sustained"],
            "peak_source": f"{peaks['source']} bf16 dense ({peak_kind}: {peak_why})",
            "kernel": ("window_assemble_kernel + mla_attn_tc_kernel<192,32,2,128> (events around both)"
                       if w.sink_frames else "mla_attn_tc_kernel<192,32,2,128>"),
            "algorithmic_flops_per_launch": attn_l,
            "traffic": (profiled_traffic("attn_tc_wan_traffic.json", "attn_tc.cu")
                        if w.batch == 1 else None),
        },
        "roofline_append": {
            "bound": "hbm", "kernel": append_kernel_name(w),
            "algorithmic_bytes_per_launch": append_bytes(w),
            "achieved": append_bytes(w) / max(app_ms, 1e-6) / 1e6,
            "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": append_bytes(w) / max(app_ms, 1e-6) / 1e6 / peaks["hbm_gbs"],
            "note": "CUDA events around each append launch (mean over a second pass of the "
                    "timed steps)",
            "back_to_back": {
                "ms": app_b2b_ms,
                "achieved": append_bytes(w) / max(app_b2b_ms, 1e-6) / 1e6,
                "frac": append_bytes(w) / max(app_b2b_ms, 1e-6) / 1e6 / peaks["hbm_gbs"],
                "note": "the timed steps' appends alone, launched back to back between two "
                        "CUDA events (mean duration per launch)",
            },
        },
        "e2e": {
            "value": tflops(attn_fl + app_fl, e2e_ms / e2e_steps),
            "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": e2e_ms / e2e_steps, "steps": e2e_steps,
            "note": "public API with pinned host buffers; every step's inputs go up and its "
                    "latent output comes back inside the timed region, on two copy streams "
                    "that overlap neighbouring layers' kernels",
        },
        "clocks": clk.summary(),
        "gpu_launches": (3 if w.sink_frames else 2) * w.layers * args.steps,
    }
    clocks = out["clocks"]
    if clocks.get("sm_mhz"):
        # the tensor pipe's own limit at the clock seen: 8192 bf16 FLOP per
        # clock per SM (our tcgen05 loops, N = 128..256, SS or TS operands)
        sms = torch.cuda.get_device_properties(0).multi_processor_count
        lim = PIPE_FLOP_PER_CLK_SM * sms * clocks["sm_mhz"] * 1e6 / 1e12
        out["roofline"]["pipe_limit_tflops"] = lim
        out["roofline"]["frac_of_pipe_limit"] = achieved / lim
    if append_b4 is not None:
        out["roofline_append_b4"] = append_b4
    if pool is not None:
        try:
            out["cpu_baseline"] = cpu_oracle_sample(w, budget_s=args.cpu_budget, pool=pool)
        finally:
            pool.close()
    return out


def time_append_b4(w, V, stream, steps=100):
    """The cache append of a 3-frame chunk at batch 4 (the rollout batch: 147
    token tiles, one per SM): launches back to back over rotating input sets
    larger than L2, timed by two CUDA events; algorithmic HBM bytes per launch
    over the mean launch duration."""
    wb = w.with_(batch=4)
    sets = []
    for i in range(N_SETS):
        wt = synth.draw_layer_weights(wb, 1500 + i)
        cache = V.LatentCache(V.make_config(wb))
        x = synth.draw_tokens(wb, wb.chunk_tokens, 1510 + i).cuda()
        pos = synth.grid_positions(wb, wb.window_frames - wb.chunk_frames, wb.chunk_frames).cuda()
        cache.frames_written = wb.window_frames
        sets.append((cache, x, wt["w_dkv"].cuda(), wt["gamma_kv"].cuda(), wt["w_kr"].cuda(), pos))
    first = wb.window_frames - wb.chunk_frames

    def launch(i):
        cache, x, wd, g, wk, pos = sets[i % N_SETS]
        V.mla_cache_append(cache, x, wd, g, wk, pos, first, wb.chunk_frames, stream)

    for i in range(5):
        launch(i)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(steps):
        launch(i)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    peaks = load_peaks()
    nbytes = append_bytes(wb)
    return {"bound": "hbm", "kernel": append_kernel_name(wb), "batch": 4,
            "algorithmic_bytes_per_launch": nbytes, "ms": ms,
            "achieved": nbytes / (ms * 1e-3) / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": nbytes / (ms * 1e-3) / 1e9 / peaks["hbm_gbs"],
            "note": f"{steps} launches back to back between two CUDA events (mean duration per "
                    f"launch), {N_SETS} rotating sets of "
                    f"{wb.chunk_tokens * 4 * w.hidden * 2 / 1e6:.0f} MB of activations"}


def run_reference(args, w):
    """The reference arm: the float64 oracle, as it stands, on every host core;
    each step is one pass over the same fixed token sample as the GPU arm's
    cpu_baseline leg."""
    pool = OraclePool(w)
    try:
        for _ in range(args.warmup):
            pool.round()
        fl = wall = cpu = 0.0
        for _ in range(args.steps):
            f, t, c = pool.round()
            fl, wall, cpu = fl + f, wall + t, cpu + c
        v = fl / wall / 1e12
        cb = {"value": v, "unit": UNIT, "cores": pool.procs,
              "cpu_utilisation": cpu / wall / pool.procs,
              "host_cores_available": len(os.sched_getaffinity(0)),
              "kind": "oracle", "sample": pool.describe(wall, args.steps), "seconds": wall}
    finally:
        pool.close()
    return {
        "impl": "reference",
        "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": 0, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": wall / max(1, args.steps) * 1e3,
        "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_desc(w)},
        "cpu_baseline": cb,
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


# ------------------------------------------------------- latent-size sweep
def time_launches(fn, steps, warmup, stream):
    """Median CUDA-event time (ms) of fn() over `steps` launches after `warmup`."""
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    ev[0].record(stream)
    for i in range(steps):
        fn()
        ev[i + 1].record(stream)
    torch.cuda.synchronize()
    return float(np.median([ev[i].elapsed_time(ev[i + 1]) for i in range(steps)]))


def run_sweep(args):
    """Latent-size sweep (the d_c axis of Table 5, left; Sec. 3.3's cache sizes):
    absorbed MLA attention for d_c in {64..512} x d_r in {32, 64} next to the
    dense per-head baseline (12 x 128 K and V per token) at the same query
    chunk and window; bytes per token, TFLOP/s and chunk latency. Shapes
    without a tensor-core instance run the SIMT kernel and say so."""
    from paper_2605_30351_gb300 import videomla as V

    V.load()
    stream = torch.cuda.current_stream()
    base = synth.workload("wan")
    peaks = load_peaks()
    layers = 30
    rows = []
    for d_c in (64, 128, 192, 256, 512):
        for d_r in (32, 64):
            pairs = (6, 5, 5) if d_r == 32 else (12, 10, 10)
            dims = (44, 42, 42) if d_r == 32 else (64, 64, 64)
            w = base.with_(d_c=d_c, d_r=d_r, rope_pairs=pairs, rope_axis_dims=dims)
            cfg = V.make_config(w)
            s = LayerSet(w, 7000 + d_c + d_r, V)
            kind = "tcgen05"
            try:
                V.mla_attention_forward(s.cache, s.q_c, s.q_r, s.pos, s.o, stream)
            except V.MlaError:
                cfg.flags = V.MLA_FLAG_SIMT
                s.cache.struct.cfg.flags = V.MLA_FLAG_SIMT
                kind = "simt (no tensor-core instance for this shape)"
            steps = args.steps if kind == "tcgen05" else 2
            ms = time_launches(lambda: V.mla_attention_forward(s.cache, s.q_c, s.q_r, s.pos, s.o,
                                                               stream), steps, 2, stream)
            fl = flops_per_layer(w)[0]
            if kind == "tcgen05" and d_c > 256:
                # the output is split over a CTA pair and both CTAs score the full key tile
                kind = "tcgen05 (output split over a CTA pair; score computed by both)"
            rows.append({
                "layout": "mla", "d_c": d_c, "d_r": d_r, "kernel": kind,
                "bytes_per_token_per_layer": 2 * (d_c + d_r),
                "cache_gb_30_layers_21_frames": layers * w.slots * (d_c + d_r) * 2 / 1e9,
                "compression_vs_dense": 2 * w.heads * w.head_dim / (d_c + d_r),
                "ms_per_chunk_layer": ms, "tflops": fl / (ms * 1e-3) / 1e12,
                "frac_of_measured_bf16_burst": fl / (ms * 1e-3) / 1e12 / peaks["bf16_tflops"],
                "flop_per_row_key": 4 * d_c + 2 * d_r,
                **({"issued_flop_per_row_key": 4 * (d_c + d_r) + 2 * d_c,
                    "issued_tflops": fl / (4 * d_c + 2 * d_r) * (4 * (d_c + d_r) + 2 * d_c)
                    / (ms * 1e-3) / 1e12} if d_c > 256 else {})})
            del s
            torch.cuda.empty_cache()
    # dense per-head baseline: q, k, v with d_h = 128, 12 heads, same window
    w = base
    cfg = V.make_config(w)
    g = torch.Generator(device="cuda").manual_seed(11)
    q = torch.randn(1, w.chunk_tokens, w.heads, w.head_dim, device="cuda", generator=g).to(torch.bfloat16)
    k = torch.randn(1, w.heads, w.slots, w.head_dim, device="cuda", generator=g).to(torch.bfloat16)
    v = torch.randn(1, w.heads, w.slots, w.head_dim, device="cuda", generator=g).to(torch.bfloat16)
    o = torch.empty_like(q)
    ms = time_launches(lambda: V.mla_dense_attention_forward(cfg, q, k, v, w.slots, o, stream),
                       args.steps, 2, stream)
    fl = 4.0 * w.chunk_tokens * w.heads * w.slots * w.head_dim
    rows.append({
        "layout": "dense", "d_h": w.head_dim, "kernel": "tcgen05",
        "bytes_per_token_per_layer": 2 * 2 * w.heads * w.head_dim,
        "cache_gb_30_layers_21_frames": layers * w.slots * 2 * w.heads * w.head_dim * 2 / 1e9,
        "ms_per_chunk_layer": ms, "tflops": fl / (ms * 1e-3) / 1e12,
        "frac_of_measured_bf16_burst": fl / (ms * 1e-3) / 1e12 / peaks["bf16_tflops"],
        "flop_per_row_key": 4 * w.head_dim})
    # decompress-then-dense on the d_c = 192 latent cache: expand every slot into
    # per-head keys [W_up^K c | k] and values W_up^V c, then the dense kernel
    s = LayerSet(base, 7300, V)
    wt = {k: t.cuda() for k, t in synth.draw_layer_weights(base, 7301).items()}
    kd = torch.empty(1, w.heads, w.slots, w.head_dim, dtype=torch.bfloat16, device="cuda")
    vd = torch.empty_like(kd)
    t_dec = time_launches(lambda: V.mla_decompress_window(s.cache, wt["w_uk"], wt["w_uv"], kd, vd,
                                                          stream), args.steps, 2, stream)
    t_att = time_launches(lambda: V.mla_dense_attention_forward(cfg, q, kd, vd, w.slots, o, stream),
                          args.steps, 2, stream)
    dn = w.head_dim - base.d_r
    fl_dec = 2.0 * w.slots * base.d_c * w.heads * (dn + w.head_dim)
    rows.append({
        "layout": "mla decompress-then-dense", "d_c": base.d_c, "d_r": base.d_r,
        "kernel": "tcgen05 (scatter GEMM + dense attention)",
        "bytes_per_token_per_layer": 2 * (base.d_c + base.d_r),
        "transient_bytes_per_layer": 2 * 2 * w.heads * w.head_dim * w.slots,
        "decompress_ms": t_dec, "attention_ms": t_att, "ms_per_chunk_layer": t_dec + t_att,
        "tflops": (fl + fl_dec) / ((t_dec + t_att) * 1e-3) / 1e12,
        "frac_of_measured_bf16_burst": (fl + fl_dec) / ((t_dec + t_att) * 1e-3) / 1e12
        / peaks["bf16_tflops"],
        "flop_per_row_key": 4 * w.head_dim,
        "decompress_flop_per_key": 2 * base.d_c * w.heads * (dn + w.head_dim)})
    if V.mla_device_status(clear=True) != V.MLA_OK:
        raise RuntimeError("device status set during the sweep")
    return {"metric": "latent-size sweep: absorbed MLA attention vs dense per-head baseline",
            "unit": "ms per chunk per layer", "data": "synthetic", "dtype": "bf16",
            "config": {"workload": workload_desc(base) + "; d_c and d_r varied"},
            "sweep": rows}


# ------------------------------------------------- the other configs, briefly
def other_configs():
    """The benchmark's other configurations, each measured in its own short
    timed region of the default run, so that one bench line covers them all:
    the tiny single layer (config 1), the 30-layer step (config 3), the batch-4
    rollout window (config 4) and the d_c x d_r sweep next to the dense
    baseline (config 5). Fewer steps than their own commands
    (`--workload tiny|wan30|rollout`, `--sweep dc`); a configuration that fails
    records its error instead of stopping the line."""
    res = {}
    for key, name, steps in (("config1_tiny", "tiny", 50), ("config3_wan30", "wan30", 5),
                             ("config4_rollout", "rollout", 20)):
        try:
            ns = argparse.Namespace(steps=steps, warmup=3, no_cpu_baseline=True, cpu_budget=0.0)
            o = run_ours(ns, synth.workload(name))
            res[key] = {"workload": o["config"]["workload"], "steps": steps,
                        "ms_per_step": o["ms_per_step"], "value": o["value"], "unit": o["unit"],
                        "attention_frac_of_peak": o["roofline"]["frac"],
                        "peak_source": o["roofline"]["peak_source"],
                        "append_frac_of_hbm": o["roofline_append"]["frac"],
                        "e2e": o["e2e"]["value"], "sm_mhz": o["clocks"].get("sm_mhz")}
        except Exception as e:  # noqa: BLE001 - recorded in the line
            res[key] = {"error": f"{type(e).__name__}: {e}"[:300]}
        torch.cuda.empty_cache()
    try:
        sw = run_sweep(argparse.Namespace(steps=10, warmup=3))
        res["config5_sweep"] = {
            "steps": 10, "unit": "ms per chunk per layer",
            "rows": [{k: r[k] for k in ("layout", "d_c", "d_r", "ms_per_chunk_layer", "tflops",
                                        "frac_of_measured_bf16_burst") if k in r}
                     for r in sw["sweep"]]}
    except Exception as e:  # noqa: BLE001
        res["config5_sweep"] = {"error": f"{type(e).__name__}: {e}"[:300]}
    torch.cuda.empty_cache()
    return res


# ------------------------------------------------------------- crossover
def run_crossover(args):
    """Absorbed attention (App. E) against decompress-then-dense (Eq.
    reconstruct, then per-head attention) as the query chunk grows from one
    latent frame to twelve, on the same 21-frame Wan window: the per-key cost
    of decompressing is paid once per window, the absorbed form's extra cost
    per (query, key)."""
    from paper_2605_30351_gb300 import videomla as V

    V.load()
    stream = torch.cuda.current_stream()
    peaks = load_peaks()
    rows = []
    for frames in (1, 2, 3, 6, 12):
        w = synth.workload("wan", chunk_frames=frames)
        nq = w.chunk_tokens
        s = LayerSet(w, 7400 + frames, V)
        wt = {k: t.cuda() for k, t in synth.draw_layer_weights(w, 7401).items()}
        t_abs = time_launches(lambda: V.mla_attention_forward(s.cache, s.q_c, s.q_r, s.pos, s.o,
                                                              stream), args.steps, 2, stream)
        cfg = s.cache.cfg
        kd = torch.empty(1, w.heads, w.slots, w.head_dim, dtype=torch.bfloat16, device="cuda")
        vd = torch.empty_like(kd)
        g = torch.Generator(device="cuda").manual_seed(frames)
        q = torch.randn(1, nq, w.heads, w.head_dim, device="cuda", generator=g).to(torch.bfloat16)
        o = torch.empty_like(q)
        t_dec = time_launches(lambda: V.mla_decompress_window(s.cache, wt["w_uk"], wt["w_uv"], kd,
                                                              vd, stream), args.steps, 2, stream)
        t_den = time_launches(lambda: V.mla_dense_attention_forward(cfg, q, kd, vd, w.slots, o,
                                                                    stream), args.steps, 2, stream)
        fl_abs = flops_per_layer(w)[0]
        rows.append({"query_frames": frames, "query_tokens": nq, "keys": w.slots,
                     "absorbed_ms": t_abs,
                     "absorbed_tflops": fl_abs / (t_abs * 1e-3) / 1e12,
                     "decompress_ms": t_dec, "dense_attention_ms": t_den,
                     "decompress_then_dense_ms": t_dec + t_den,
                     "absorbed_over_decompressed": t_abs / (t_dec + t_den)})
        del s, kd, vd, q, o
        torch.cuda.empty_cache()
    if V.mla_device_status(clear=True) != V.MLA_OK:
        raise RuntimeError("device status set during the crossover sweep")
    return {"metric": "absorbed MLA attention vs decompress-then-dense, by query-chunk size",
            "unit": "ms per chunk per layer", "data": "synthetic", "dtype": "bf16",
            "peak_bf16_tflops": peaks["bf16_tflops"],
            "config": {"workload": "Wan2.1-1.3B layer: 21-frame window (32,760 keys), 12 heads, "
                                   "d_c=192, d_r=32, batch 1; query chunk of 1..12 latent frames"},
            "crossover": rows}


# ------------------------------------------------------------- full layer
def run_layer(args, w):
    """The whole attention layer per chunk (Sec. 3, App. E): query prologue
    (x -> c^Q -> RMSNorm -> [q_c | q_r], absorbed weights), cache append,
    latent attention and output projection y = sum_h B_h o_lat,h; each phase
    timed with CUDA events, inputs rotating over layer sets larger than L2."""
    from paper_2605_30351_gb300 import videomla as V

    V.load()
    stream = torch.cuda.current_stream()
    nq = w.chunk_tokens
    sets = []
    for i in range(N_SETS):
        s = LayerSet(w, 1200 + 17 * i, V)
        wt = {k: t.cuda() for k, t in synth.draw_layer_weights(w, 1200 + 17 * i).items()}
        cfg = s.cache.cfg
        s.w_dq = wt["w_dq"]
        s.w_qcat, s.w_b = V.mla_absorb_weights(cfg, wt["w_uq"], wt["w_uk"], wt["w_qr"],
                                               wt["gamma_q"], wt["w_uv"], wt["w_o"])
        s.ws_q = torch.empty(V.mla_query_workspace_bytes(cfg, nq), dtype=torch.uint8, device="cuda")
        s.y = torch.empty(w.batch, nq, w.hidden, dtype=torch.bfloat16, device="cuda")
        sets.append(s)

    def layer(s, ev=None):
        cfg = s.cache.cfg
        if ev is not None:
            ev[0].record(stream)
        V.mla_query_prologue(cfg, s.x, s.w_dq, s.w_qcat, s.ws_q, s.q_c, s.q_r, stream)
        if ev is not None:
            ev[1].record(stream)
        V.mla_cache_append(s.cache, s.x, s.w_dkv, s.gamma, s.w_kr, None if s.window else s.pos,
                           s.first, w.chunk_frames, stream)
        if ev is not None:
            ev[2].record(stream)
        if s.window:
            V.mla_attention_window_forward(s.cache, s.q_c, s.q_r, s.pos, s.hw, s.ws, s.o, stream)
        else:
            V.mla_attention_forward(s.cache, s.q_c, s.q_r, s.pos, s.o, stream)
        if ev is not None:
            ev[3].record(stream)
        V.mla_output_projection(cfg, s.o, s.w_b, s.y, stream)
        if ev is not None:
            ev[4].record(stream)

    for i in range(max(3, args.warmup)):
        layer(sets[i % N_SETS])
    torch.cuda.synchronize()
    steps = max(1, args.steps)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(steps)]
    for i in range(steps):
        layer(sets[i % N_SETS], evs[i])
    torch.cuda.synchronize()
    if V.mla_device_status(clear=True) != V.MLA_OK:
        raise RuntimeError("device status set during the layer timing")
    med = [float(np.median([e[k].elapsed_time(e[k + 1]) for e in evs])) for k in range(4)]
    total = float(np.median([e[0].elapsed_time(e[4]) for e in evs]))
    rows = w.batch * nq
    attn_fl, app_fl = flops_per_layer(w)
    pro_fl = 2.0 * rows * w.hidden * w.d_q + 2.0 * rows * w.d_q * w.heads * (w.d_c + w.d_r)
    out_fl = 2.0 * rows * w.heads * w.d_c * w.hidden
    peaks = load_peaks()
    phases = {}
    for name, ms, fl in (("query_prologue", med[0], pro_fl), ("append", med[1], app_fl),
                         ("attention", med[2], attn_fl), ("output_projection", med[3], out_fl)):
        phases[name] = {"ms": ms, "flop": fl, "tflops": fl / (ms * 1e-3) / 1e12,
                        "frac_of_measured_bf16_burst": fl / (ms * 1e-3) / 1e12 / peaks["bf16_tflops"]}
    fl_all = pro_fl + app_fl + attn_fl + out_fl
    return {"metric": "full attention layer per chunk: prologue, append, attention, output projection",
            "value": fl_all / (total * 1e-3) / 1e12, "unit": "TFLOP/s", "ms_per_layer": total,
            "higher_is_better": True, "data": "synthetic", "dtype": "bf16", "steps": steps,
            "config": {"workload": workload_desc(w).replace(
                "step = cache append + attention", "step = query prologue + cache append + "
                "attention + output projection"),
                       "l2": f"{N_SETS} rotating layer sets"},
            "phases": phases, "gpu_launches_per_layer": 5 + (1 if w.sink_frames else 0)}


# ------------------------------------------------------ memory-cap batch sweep
B200_USABLE_GB = 180.0  # HBM of the B200 the paper's batch-scaling figure ran on


def memcap_plan(w, layout, budget_bytes, layers=30):
    """Largest batch whose attention-path state fits in `budget_bytes` (Sec. 4,
    batch scaling under fixed memory: the caches decide when MHA runs out).

    Per batch element: the caches of every layer for the whole window
    (`layout` "mla": c and k_r, 2 (d_c + d_r) bytes per token per layer;
    "dense": per-head K and V, 2 * 2 * H * d_h) plus one layer's chunk
    activations in flight (x, positions, queries, attention output, y). Fixed:
    every layer's projection weights. The rest of the DiT (FFN, norms) is not
    counted."""
    n, hid, H = w.chunk_tokens, w.hidden, w.heads
    if layout == "mla":
        cache_tok = 2 * (w.d_c + w.d_r)
        q_row, o_row = H * (w.d_c + w.d_r) * 2, H * w.d_c * 2
        weights = 2 * ((w.d_c + w.d_r) * hid + w.d_c + w.d_q * hid + w.d_q
                       + H * (w.d_c + w.d_r) * w.d_q + hid * H * w.d_c)
    else:
        cache_tok = 2 * 2 * H * w.head_dim
        q_row, o_row = H * w.head_dim * 2, H * w.head_dim * 2
        weights = 2 * 4 * hid * H * w.head_dim
    cache_b = layers * w.slots * cache_tok
    act_b = n * (hid * 2 + 3 * 4 + q_row + o_row + hid * 2)
    per_batch = cache_b + act_b
    fixed = layers * weights
    b_max = max(0, int((budget_bytes - fixed) // per_batch))
    return {"cache_bytes_per_batch": cache_b, "activation_bytes_per_batch": act_b,
            "weight_bytes": fixed, "per_batch_bytes": per_batch, "max_batch": b_max,
            "bytes_at_max_batch": fixed + b_max * per_batch}


def run_memcap(args):
    """Maximum batch of one chunk-against-window attention step under a fixed
    HBM budget, dense per-head caches against latent caches at several d_c;
    the plan is checked by allocating every layer's cache at that batch and
    running one layer there (append and attention for the latent layout,
    attention for the dense one)."""
    from paper_2605_30351_gb300 import videomla as V

    V.load()
    stream = torch.cuda.current_stream()
    base = synth.workload("wan")
    layers = 30
    budget = args.mem_budget_gb * 1e9
    total = torch.cuda.mem_get_info()[1]
    layouts = [("dense", base)] + [("mla", base.with_(d_c=dc)) for dc in (64, 128, 192, 256, 512)]
    rows = []
    g = torch.Generator(device="cuda").manual_seed(23)
    for layout, w in layouts:
        plan = memcap_plan(w, layout, budget, layers)
        whole = memcap_plan(w, layout, total - 4e9, layers)
        B = plan["max_batch"]
        wb = w.with_(batch=B)
        row = {"layout": layout, "d_c": w.d_c if layout == "mla" else None,
               "d_r": w.d_r if layout == "mla" else None,
               "gb_per_batch": plan["per_batch_bytes"] / 1e9,
               "cache_gb_per_batch": plan["cache_bytes_per_batch"] / 1e9,
               "max_batch": B, f"max_batch_{total / 1e9:.0f}gb_device": whole["max_batch"]}
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        before = torch.cuda.memory_allocated()
        nq = w.chunk_tokens
        if layout == "mla":
            cfg = V.make_config(wb)
            caches = [V.LatentCache(cfg) for _ in range(layers)]
            x = torch.empty(B, nq, w.hidden, dtype=torch.bfloat16, device="cuda")
            pos = torch.empty(B, nq, 3, dtype=torch.int32, device="cuda")
            q_c = torch.empty(B, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
            q_r = torch.empty(B, nq, w.heads, w.d_r, dtype=torch.bfloat16, device="cuda")
            o = torch.empty(B, nq, w.heads, w.d_c, dtype=torch.bfloat16, device="cuda")
            y = torch.empty(B, nq, w.hidden, dtype=torch.bfloat16, device="cuda")
            wt = {k: v.cuda() for k, v in synth.draw_layer_weights(w, 29).items()}
        else:
            kv = [(torch.empty(B, w.heads, w.slots, w.head_dim, dtype=torch.bfloat16, device="cuda"),
                   torch.empty(B, w.heads, w.slots, w.head_dim, dtype=torch.bfloat16, device="cuda"))
                  for _ in range(layers)]
            x = torch.empty(B, nq, w.hidden, dtype=torch.bfloat16, device="cuda")
            q = torch.empty(B, nq, w.heads, w.head_dim, dtype=torch.bfloat16, device="cuda")
            o = torch.empty_like(q)
            y = torch.empty_like(x)
        used = torch.cuda.memory_allocated() - before
        row["allocated_gb_at_max_batch"] = used / 1e9
        row["fits_budget"] = bool(used <= budget)
        fl_row = (4 * w.d_c + 2 * w.d_r) if layout == "mla" else 4 * w.head_dim
        fl = 1.0 * B * nq * w.heads * w.slots * fl_row
        tc = layout == "dense" or (w.d_c, w.d_r) in ((64, 32), (128, 32), (192, 32), (256, 32),
                                                     (512, 32))
        if B > 0 and tc:
            if layout == "mla":
                c0 = caches[0]
                c0.c.normal_(generator=g)
                c0.kr.normal_(generator=g)
                c0.frames_written = w.window_frames
                x.normal_(generator=g)
                q_c.normal_(generator=g)
                q_r.normal_(generator=g)
                pos.copy_(synth.grid_positions(wb, w.window_frames - w.chunk_frames,
                                               w.chunk_frames).to(pos.device))
                first = w.window_frames - w.chunk_frames
                t_app = time_launches(lambda: V.mla_cache_append(
                    c0, x, wt["w_dkv"], wt["gamma_kv"], wt["w_kr"], pos, first, w.chunk_frames,
                    stream), 3, 1, stream)
                t_att = time_launches(lambda: V.mla_attention_forward(c0, q_c, q_r, pos, o, stream),
                                      3, 1, stream)
                row["append_ms_at_max_batch"] = t_app
            else:
                k0, v0 = kv[0]
                k0.normal_(generator=g)
                v0.normal_(generator=g)
                q.normal_(generator=g)
                cfg = V.make_config(wb)
                t_att = time_launches(lambda: V.mla_dense_attention_forward(cfg, q, k0, v0, w.slots,
                                                                            o, stream), 3, 1, stream)
            row["attention_ms_at_max_batch"] = t_att
            row["attention_tflops_at_max_batch"] = fl / (t_att * 1e-3) / 1e12
            row["query_tokens_per_s_one_layer"] = B * nq / (t_att * 1e-3)
            status = V.mla_device_status(clear=True)
            if status != V.MLA_OK:
                raise RuntimeError(f"device status {status} in the memory-cap run")
        else:
            row["attention_ms_at_max_batch"] = None
            row["note"] = "allocation only: no tensor-core instance for this shape"
        rows.append(row)
        del x, o, y
        if layout == "mla":
            del caches, q_c, q_r, pos, wt
        else:
            del kv, q
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
    return {"metric": "maximum batch under a fixed HBM budget: dense per-head vs latent caches",
            "unit": "batch elements (one 4680-token chunk against a 21-frame window each)",
            "data": "synthetic", "dtype": "bf16",
            "config": {"workload": workload_desc(base) + f"; {layers} layers of caches; budget "
                       f"{args.mem_budget_gb:g} GB (a B200's usable HBM) and the whole device"},
            "memcap": rows}


# ----------------------------------------------------------------- helpers
PIPE_FLOP_PER_CLK_SM = 8192  # measured tcgen05 bf16 rate per SM (N = 128..256)
MULTI_GPU_CLOSED = ("multi-GPU runs are closed on this pool: the attention kernels share key "
                    "tiles among the CTAs of a cluster by TMA multicast, which may only run in "
                    "single-GPU jobs")


def tflops(flop_per_step, ms_per_step):
    return flop_per_step / (ms_per_step * 1e-3) / 1e12


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="wan")
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", choices=["dc", "memcap", "layer", "crossover"], default=None,
                    help="dc: latent-size sweep next to the dense baseline; memcap: maximum "
                         "batch under --mem-budget-gb; layer: the whole attention layer by "
                         "phase; crossover: absorbed vs decompress-then-dense by chunk size "
                         "(one JSON line each)")
    ap.add_argument("--mem-budget-gb", type=float, default=B200_USABLE_GB)
    ap.add_argument("--no-other-configs", action="store_true",
                    help="skip the brief measurements of configs 1, 3, 4 and 5 that the "
                         "default run adds to its line")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    w = synth.workload(args.workload)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if world > 1 or args.gpus > 1:
        # no multi-GPU path (see the module docstring); rank 0 reports, every
        # rank exits 0 without touching a GPU
        if rank != 0:
            return
        if args.impl == "reference":
            out = run_reference(args, w)
        else:
            out = {"metric": METRIC, "unit": UNIT, "n_gpus": max(world, args.gpus),
                   "unavailable": MULTI_GPU_CLOSED}
        print(json.dumps(out), flush=True)
        return
    if args.sweep == "dc":
        out = run_sweep(args)
    elif args.sweep == "memcap":
        out = run_memcap(args)
    elif args.sweep == "layer":
        out = run_layer(args, w)
    elif args.sweep == "crossover":
        out = run_crossover(args)
    elif args.impl == "reference":
        out = run_reference(args, w)
    else:
        out = run_ours(args, w)
        if args.workload == "wan" and not args.no_other_configs:
            out["other_configs"] = other_configs()
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()

"""Benchmark of one MBE editing pass on synthetic decoding-shaped data.

A step is one editing pass of the whole hot path over one batch: window
attention for every layer (one mbe_window_attention call per layer) followed
by mbe_edit_decide over the pass's logits; workloads that include the cache
refresh also run mbe_kv_window_write. Inputs are resident in HBM when the timed
region starts. The default workload is the decode-heavy serving mix
(128 sequences, prefix U[512,16384], window 64, 32/8 heads, head_dim 128,
24 layers, vocabulary 131072).

Prints one JSON line (rank 0). ``--impl reference`` times the CPU oracle on a
bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "edit-pass attn TFLOP/s (% bf16 peak); edit-decide GB/s (% HBM); windows/s"
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in PEAKS_FALLBACK}, "measured"
    except Exception:
        return dict(PEAKS_FALLBACK), "fallback"


# ------------------------------------------------------------------ accounting
def attention_flops(prefix, window, modes, num_q_heads, head_dim, block_size):
    """Mask-aware algorithmic FLOPs: 4 * D per visible (query, key) pair and
    query head (QK^T and PV, one multiply-add = 2 FLOPs each)."""
    pairs = 0
    for P, W, m in zip(prefix, window, modes):
        if m == 1:
            pairs += W * (P + W)
        else:
            for i in range(W):
                pairs += P + min(W, (i // block_size + 1) * block_size)
    return 4 * head_dim * num_q_heads * pairs


def attention_bytes(prefix, window, num_q_heads, num_kv_heads, head_dim):
    """Algorithmic HBM bytes: each prefix and window K/V row read once, Q read
    once, O written once (bf16)."""
    kv = sum(P + W for P, W in zip(prefix, window)) * num_kv_heads * head_dim * 2 * 2
    qo = sum(window) * num_q_heads * head_dim * 2 * 2
    return kv + qo


def edit_bytes(rows, vocab, elem):
    """Logits read once + committed read + new token, mask, confidence written."""
    return rows * vocab * elem + rows * (4 + 4 + 1 + 4)


# ------------------------------------------------------------------ measured traffic
# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) of one attention call
# (attn_kernel) of the serving workload, keyed by the first 16 hex digits of the
# SHA-256 of the kernel source that was measured; a changed kernel gets no traffic
# figure until it is measured again. Measured on a 64-sequence, one-layer case of
# the same workload (2.3 GB of cache on the device), whose reads were 1.0092x its
# algorithmic Q + K/V bytes; scaled to the 128-sequence call by those bytes, plus
# its output (the full call splits no key range, so it writes no partials).
# Source: profiles/attn_kernel_dram_serving_b64.md.
MEASURED_TRAFFIC = {
    "d2f0654adf59f35a": {"serving128": 4436701626 + 67108864},
}


def measured_traffic(workload):
    import hashlib
    try:
        with open(os.path.join(ROOT, "paper_2607_22663_gb300", "csrc", "attention.cu"), "rb") as f:
            h = hashlib.sha256(f.read()).hexdigest()[:16]
    except OSError:
        return None
    return MEASURED_TRAFFIC.get(h, {}).get(workload)


# ------------------------------------------------------------------ ranks
def max_over_ranks(x: float, device="cpu") -> float:
    """Maximum of a per-rank scalar over all ranks (identity on one rank)."""
    if not torch.distributed.is_available() or not torch.distributed.is_initialized():
        return x
    if torch.distributed.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: int, world: int, seconds_max: float) -> float:
    """Units processed by all ranks per second of the slowest rank."""
    return units_per_rank * world / seconds_max


# ------------------------------------------------------------------ clocks
class ClockSampler:
    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
            os.unlink(self.path)
        except Exception:
            pass
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows)}


# ------------------------------------------------------------------ workloads
def build_workload(name, device, layers=None, batch=None, vocab=None):
    from paper_2607_22663_gb300 import workloads as wl
    if name == "serving128":
        return wl.serving128(device, layers=layers or 24, batch=batch or 128, vocab=vocab or 131072)
    return wl.WORKLOADS[name](device)


def workload_config(w):
    a = w["attn"][0]
    cfg = {"workload": w["name"], "batch": a.batch, "layers": w["layers"], "attn_calls_per_step": len(w["attn"]),
           "window": sorted(set(a.window_host)), "prefix_range": [min(a.prefix_host), max(a.prefix_host)],
           "heads_q_kv": [a.num_q_heads, a.num_kv_heads], "head_dim": a.head_dim, "block_size": a.block_size,
           "page_size": a.page_size}
    if w.get("edit") is not None:
        cfg["edit_rows_vocab"] = list(w["edit"].logits.shape)
    return cfg


# ------------------------------------------------------------------ GPU arm
def run_gpu(args, rank, world):
    from paper_2607_22663_gb300 import mbe
    from paper_2607_22663_gb300.workloads import editable_historical

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    peaks, peak_src = load_peaks()
    w = build_workload(args.workload, dev, args.layers, args.batch, args.vocab)
    attn = w["attn"]
    ep = w["edit"]
    with_kv_write = args.workload == "long32k"
    a0 = attn[0]
    editable = editable_historical(a0.window_host, a0.block_size, dev) if ep is not None else None
    stream = torch.cuda.current_stream()

    # per-call buffers: outputs, workspaces and per-call events
    outs = [torch.empty_like(a.q) for a in attn]
    # one workspace serves every call: the calls run in order on one stream
    need = max(mbe.window_attention_workspace_size(a.batch, a.num_q_heads, a.num_kv_heads, a.head_dim, a.max_window,
                                                   a.max_prefix) for a in attn)
    ws = torch.empty(need, dtype=torch.uint8, device=dev)
    wss = [ws] * len(attn)
    if ep is not None:
        R = ep.logits.shape[0]
        new_t = torch.empty(R, dtype=torch.int32, device=dev)
        mask_t = torch.empty(R, dtype=torch.uint8, device=dev)
        conf_t = torch.empty(R, dtype=torch.float32, device=dev)

    # one plan per pass when every call shares the lengths, modes and bounds
    plan_layers = len({(id(a.prefix_len), id(a.window_len), id(a.cu_window), id(a.mask_mode), a.max_window,
                        a.max_prefix, a.total_tokens) for a in attn}) == 1

    def attention_call(i, a, q=None, kw=None, vw=None):
        # the first call of a pass plans (mbe_window_attention = plan + run); the
        # other layers reuse that work list
        fn = mbe.window_attention if (i == 0 or not plan_layers) else mbe.window_attention_run
        fn(a.q if q is None else q, a.k_win if kw is None else kw, a.v_win if vw is None else vw,
           a.k_cache, a.v_cache, a.block_table, a.prefix_len, a.window_len, a.cu_window,
           a.mask_mode, block_size=a.block_size, max_window=a.max_window, max_prefix=a.max_prefix,
           out=outs[i], workspace=wss[i])

    def edit_call(logits=None, committed=None):
        mbe.edit_decide(ep.logits if logits is None else logits, ep.committed if committed is None else committed,
                        tau=ep.tau, tau_per_row=ep.tau_per_row, editable=editable, new_tokens=new_t,
                        edit_mask=mask_t, confidence=conf_t, want_argmax=False)

    def step(attn_events=None, edit_events=None):
        for i, a in enumerate(attn):
            if attn_events is not None:
                attn_events[i][0].record(stream)
            attention_call(i, a)
            if attn_events is not None:
                attn_events[i][1].record(stream)
            if with_kv_write:
                mbe.kv_window_write(a.k_win, a.v_win, a.k_cache, a.v_cache, a.block_table, a.prefix_len,
                                    a.window_len, a.cu_window, block_size=a.block_size, max_window=a.max_window)
        if ep is not None:
            if edit_events is not None:
                edit_events[0].record(stream)
            edit_call()
            if edit_events is not None:
                edit_events[1].record(stream)

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    for _ in range(args.warmup):
        step()
    st, flags = mbe.get_device_error()
    if st != 0:
        raise RuntimeError(f"device error during warm-up: status {st} flags {flags:#x}")

    K = args.steps
    ev_attn = [[[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in attn] for _ in range(K)]
    ev_edit = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(dev.index) as clk:
        barrier()
        t0.record(stream)
        for k in range(K):
            step(ev_attn[k], ev_edit[k] if ep is not None else None)
        t1.record(stream)
        barrier()
    clocks = clk.summary()
    ms_total = max_over_ranks(t0.elapsed_time(t1), dev)
    ms_step = ms_total / K
    attn_ms = [statistics.mean(ev_attn[k][i][0].elapsed_time(ev_attn[k][i][1]) for k in range(K))
               for i in range(len(attn))]
    edit_ms = statistics.mean(ev_edit[k][0].elapsed_time(ev_edit[k][1]) for k in range(K)) if ep is not None else None
    st, flags = mbe.get_device_error()
    if st != 0:
        raise RuntimeError(f"device error during timing: status {st} flags {flags:#x}")

    flops = [attention_flops(a.prefix_host, a.window_host, a.mode_host, a.num_q_heads, a.head_dim, a.block_size)
             for a in attn]
    abytes = [attention_bytes(a.prefix_host, a.window_host, a.num_q_heads, a.num_kv_heads, a.head_dim) for a in attn]
    attn_time = sum(attn_ms)
    attn_tflops = sum(flops) / (attn_time * 1e-3) / 1e12
    attn_gbs = sum(abytes) / (attn_time * 1e-3) / 1e9
    value = whole_job_rate(a0.batch, world, ms_step * 1e-3)
    res = {"metric": METRIC, "value": round(value, 3), "unit": "windows/s", "n_gpus": world, "steps": K,
           "warmup": args.warmup, "ms_per_step": round(ms_step, 4), "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
           "config": {**workload_config(w), "l2": "inputs larger than L2 (per-layer KV cache and logits >> 129 MB)",
                      "parallelism": f"replicas{world}"}}
    res["attention"] = {"tflops": round(attn_tflops, 2),
                        "frac_bf16_peak_sustained": round(attn_tflops / peaks["bf16_tflops_sustained"], 4),
                        "frac_bf16_peak_burst": round(attn_tflops / peaks["bf16_tflops"], 4),
                        "gbs": round(attn_gbs, 1), "frac_hbm": round(attn_gbs / peaks["hbm_gbs"], 4),
                        "ms_per_call": round(attn_time / len(attn), 4), "flops_per_call": flops[0],
                        "bytes_per_call": abytes[0]}
    if ep is not None:
        eb = edit_bytes(ep.logits.shape[0], ep.logits.shape[1], ep.logits.element_size())
        res["edit_decide"] = {"gbs": round(eb / (edit_ms * 1e-3) / 1e9, 1),
                              "frac_hbm": round(eb / (edit_ms * 1e-3) / 1e9 / peaks["hbm_gbs"], 4),
                              "ms": round(edit_ms, 4), "bytes": eb,
                              "edit_rate": round(float(mask_t.float().mean().item()), 5)}
    res["roofline"] = {"bound": "hbm", "achieved": round(attn_gbs, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                       "frac": round(attn_gbs / peaks["hbm_gbs"], 4), "traffic": measured_traffic(args.workload) if args.batch in (None, 128) else None,
                       "kernel": "mbe_window_attention per layer (attn_kernel + split merge; one plan per pass)",
                       "peak_source": f"{peak_src} hbm_gbs"}
    res["clocks"] = clocks
    per_step = len(attn) * 2 + (1 if plan_layers else len(attn)) + (1 if ep is not None else 0) + \
        (len(attn) if with_kv_write else 0)
    res["gpu_launches"] = per_step * K
    if args.no_extras:
        return res
    # end to end first, on the state the timed loop left (the extras allocate large buffers of their own)
    res["e2e"] = run_e2e(args, w, attention_call, edit_call, dev, stream, world, new_t if ep is not None else None,
                         mask_t if ep is not None else None, conf_t if ep is not None else None)
    if ep is not None:
        res["extras"] = time_extras(w, a0, dev, stream, peaks)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        v, desc, spent = run_cpu_sample(w, target_s=15.0)
        res["cpu_baseline"] = {"value": round(v, 5), "unit": "windows/s", "cores": oracle.num_threads(),
                               "kind": "oracle", "sample": desc}
    return res


def time_denoise_select(w, a0, dev, peaks, ev_time):
    """The full Eq. 2 update of a standard decoding step over the pass's logits (a
    third of the rows masked) and the tail-entropy window choice for every sequence."""
    from paper_2607_22663_gb300 import mbe
    ep = w["edit"]
    R, V = ep.logits.shape
    mask_id = V - 1
    tokens = ep.committed.clone()
    tokens[torch.arange(R, device=dev) % 3 == 0] = mask_id
    # max_blocks from the host-side window lengths and the outputs of a first call
    # reused, as in a captured pass: the timed calls hold no host synchronisation
    B = a0.block_size
    kw = dict(block_size=B, mask_id=mask_id, omega_mask=0.5, omega_edit=0.0)
    out = mbe.denoise_update(ep.logits, tokens, a0.cu_window, max_blocks=(max(a0.window_host) + B - 1) // B, **kw)
    ms = ev_time(lambda: mbe.denoise_update(ep.logits, tokens, a0.cu_window, out=out, **kw))
    byts = R * V * ep.logits.element_size() + R * (4 + 4 + 1 + 4 + 4 + 4)
    ent = torch.rand(a0.batch, 3, a0.block_size, device=dev)
    nv = torch.full((a0.batch,), 3, dtype=torch.int32, device=dev)
    ms_sel = ev_time(lambda: mbe.tail_entropy_select(ent, nv, rho=0.25, k_max=4))
    return {"denoise_update": {"ms": round(ms, 4), "gbs": round(byts / (ms * 1e-3) / 1e9, 1),
                               "frac_hbm": round(byts / (ms * 1e-3) / 1e9 / peaks["hbm_gbs"], 4),
                               "rows": R, "vocab": V},
            "tail_entropy_select": {"us": round(ms_sel * 1e3, 2), "sequences": a0.batch, "k_max": 4, "rho": 0.25}}


def time_extras(w, a0, dev, stream, peaks, reps=10):
    """Entry points around the editing pass, timed outside the step: the full Eq. 2
    update and the tail-entropy choice, the other workloads, the fused LM head, the
    SFT attention, the targeted refresh and the graph pass loop."""
    from paper_2607_22663_gb300 import mbe

    def ev_time(fn):
        for _ in range(3):
            fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    denoise = time_denoise_select(w, a0, dev, peaks, ev_time)
    workloads = time_workloads(dev, stream, peaks)
    lm_head = time_lm_head(w, dev, peaks, ev_time)
    sft = time_sft_attention(dev, peaks, ev_time)
    refresh = time_refresh(w, dev, stream, peaks, ev_time)
    loop = time_pass_loop(w, dev, reps=3)
    st, flags = mbe.get_device_error()
    if st != 0:
        raise RuntimeError(f"device error in extras: status {st} flags {flags:#x}")
    return {**denoise, "lm_head_edit_decide": lm_head, "sft_attention": sft, "refresh": refresh,
            "pass_loop": loop, **workloads}


def time_workloads(dev, stream, peaks, reps=10):
    """Device-timed attention of the other workloads, one block each:
    long32k (long-context editing: windows of 64, 128 and 256 queries over a
    32768-token prefix, each call followed by the window's KV write), varlen64
    (64 sequences of mixed window sizes and both mask modes, plus its edit
    decision) and batch8 (8 uniform sequences). Every attention call plans and
    runs (mbe_window_attention), as a one-layer pass does. Inputs larger than
    L2, except batch8, for which a 256 MiB buffer is written before every call;
    only the calls themselves lie between their CUDA events."""
    from paper_2607_22663_gb300 import mbe
    from paper_2607_22663_gb300 import workloads as wl
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    res = {}
    for name in ("long32k", "varlen64", "batch8"):
        w = wl.WORKLOADS[name](dev)
        calls, ep = w["attn"], w["edit"]
        with_kv_write = name == "long32k"
        need = max(mbe.window_attention_workspace_size(a.batch, a.num_q_heads, a.num_kv_heads, a.head_dim,
                                                       a.max_window, a.max_prefix) for a in calls)
        ws = torch.empty(need, dtype=torch.uint8, device=dev)
        outs = [torch.empty_like(a.q) for a in calls]
        abytes = [attention_bytes(a.prefix_host, a.window_host, a.num_q_heads, a.num_kv_heads, a.head_dim)
                  for a in calls]
        flops = [attention_flops(a.prefix_host, a.window_host, a.mode_host, a.num_q_heads, a.head_dim, a.block_size)
                 for a in calls]
        small = max(abytes) < 2 * 129e6

        def attend(i, a):
            mbe.window_attention(a.q, a.k_win, a.v_win, a.k_cache, a.v_cache, a.block_table, a.prefix_len,
                                 a.window_len, a.cu_window, a.mask_mode, block_size=a.block_size,
                                 max_window=a.max_window, max_prefix=a.max_prefix, out=outs[i], workspace=ws)

        def write(a):
            mbe.kv_window_write(a.k_win, a.v_win, a.k_cache, a.v_cache, a.block_table, a.prefix_len, a.window_len,
                                a.cu_window, block_size=a.block_size, max_window=a.max_window)

        ev = [[[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in calls] for _ in range(reps + 3)]
        for r in range(reps + 3):
            for i, a in enumerate(calls):
                if small:
                    flush.fill_(r & 0xFF)
                ev[r][i][0].record(stream)
                attend(i, a)
                ev[r][i][1].record(stream)
                if with_kv_write:
                    write(a)
                ev[r][i][2].record(stream)
        torch.cuda.synchronize()
        ms = [statistics.mean(ev[r][i][0].elapsed_time(ev[r][i][1]) for r in range(3, reps + 3))
              for i in range(len(calls))]
        t = sum(ms) * 1e-3
        tf = sum(flops) / t / 1e12
        gbs = sum(abytes) / t / 1e9
        blk = {"attention_ms_per_call": [round(x, 4) for x in ms], "window": [a.max_window for a in calls],
               "attention_tflops": round(tf, 1), "frac_bf16_peak_sustained": round(tf / peaks["bf16_tflops_sustained"], 4),
               "frac_bf16_peak_burst": round(tf / peaks["bf16_tflops"], 4), "attention_gbs": round(gbs, 1),
               "frac_hbm": round(gbs / peaks["hbm_gbs"], 4), "flops": flops, "bytes": abytes,
               "l2": "256 MiB written before each call" if small else "inputs larger than L2",
               "config": workload_config(w)}
        if with_kv_write:
            kv_ms = [statistics.mean(ev[r][i][1].elapsed_time(ev[r][i][2]) for r in range(3, reps + 3))
                     for i in range(len(calls))]
            kv_bytes = [2 * 2 * sum(a.window_host) * a.num_kv_heads * a.head_dim * 2 for a in calls]
            blk["kv_write_ms_per_call"] = [round(x, 4) for x in kv_ms]
            blk["kv_write_gbs"] = [round(b / (x * 1e-3) / 1e9, 1) for b, x in zip(kv_bytes, kv_ms)]
            blk["windows_per_s"] = round(calls[0].batch * len(calls) / ((sum(ms) + sum(kv_ms)) * 1e-3), 1)
        if ep is not None:
            new = torch.empty(ep.logits.shape[0], dtype=torch.int32, device=dev)
            msk = torch.empty_like(new, dtype=torch.uint8)
            cf = torch.empty_like(new, dtype=torch.float32)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            tot = 0.0
            for r in range(reps + 3):
                if small:
                    flush.fill_(r & 0xFF)
                e0.record(stream)
                mbe.edit_decide(ep.logits, ep.committed, tau=ep.tau, tau_per_row=ep.tau_per_row, new_tokens=new,
                                edit_mask=msk, confidence=cf, want_argmax=False)
                e1.record(stream)
                torch.cuda.synchronize()
                if r >= 3:
                    tot += e0.elapsed_time(e1)
            ems = tot / reps
            eb = edit_bytes(ep.logits.shape[0], ep.logits.shape[1], ep.logits.element_size())
            blk["edit_decide"] = {"ms": round(ems, 4), "gbs": round(eb / (ems * 1e-3) / 1e9, 1),
                                  "frac_hbm": round(eb / (ems * 1e-3) / 1e9 / peaks["hbm_gbs"], 4)}
            blk["windows_per_s"] = round(calls[0].batch / ((sum(ms) + ems) * 1e-3), 1)
        elif not with_kv_write:
            blk["windows_per_s"] = round(calls[0].batch / t, 1)
        res[name] = blk
        del w, calls, ep, ws, outs
        torch.cuda.empty_cache()
    del flush
    return res


def time_lm_head(w, dev, peaks, ev_time, hidden=4096):
    """LM-head projection fused with the edit decision (the logits never reach
    HBM) on random weights, against cuBLAS writing bf16 logits followed by the
    HBM-streaming edit decision."""
    from paper_2607_22663_gb300 import mbe
    ep = w["edit"]
    R, V = ep.logits.shape
    g = torch.Generator(device=dev).manual_seed(123)
    h = torch.randn(R, hidden, generator=g, device=dev).to(torch.bfloat16)
    W = (torch.randn(V, hidden, generator=g, device=dev) * (2.0 / hidden ** 0.5)).to(torch.bfloat16)
    ws = torch.empty(mbe.lm_head_workspace_size(R, V), dtype=torch.uint8, device=dev)
    new = torch.empty(R, dtype=torch.int32, device=dev)
    mask = torch.empty(R, dtype=torch.uint8, device=dev)
    conf = torch.empty(R, dtype=torch.float32, device=dev)
    fused = ev_time(lambda: mbe.lm_head_edit_decide(h, W, ep.committed, tau=ep.tau, new_tokens=new, edit_mask=mask,
                                                    confidence=conf, want_argmax=False, workspace=ws))
    logits = torch.empty(R, V, dtype=torch.bfloat16, device=dev)
    gemm = ev_time(lambda: torch.matmul(h, W.t(), out=logits))

    def unfused():
        torch.matmul(h, W.t(), out=logits)
        mbe.edit_decide(logits, ep.committed, tau=ep.tau, new_tokens=new, edit_mask=mask, confidence=conf,
                        want_argmax=False)
    unf = ev_time(unfused)
    flops = 2.0 * R * V * hidden
    tf = flops / (fused * 1e-3) / 1e12
    del logits, W, h
    return {"ms": round(fused, 4), "tflops": round(tf, 1), "frac_bf16_peak_burst": round(tf / peaks["bf16_tflops"], 4),
            "frac_bf16_peak_sustained": round(tf / peaks["bf16_tflops_sustained"], 4), "rows": R, "vocab": V,
            "hidden": hidden, "cublas_gemm_ms": round(gemm, 4),
            "cublas_tflops": round(flops / (gemm * 1e-3) / 1e12, 1), "cublas_gemm_plus_edit_decide_ms": round(unf, 4),
            "note": "random bf16 weights; roofline bound: tensor"}


def time_sft_attention(dev, peaks, ev_time, batch=4, n_prompt=4, n_blocks=64, K=4, B=32):
    """Multi-Block Edit SFT attention (Sec. 3) on a seeded training batch: the
    cross-block mask, the forward and the backward; FLOPs count visible token
    pairs only (4 D Hq per pair forward, 10 D Hq backward)."""
    from paper_2607_22663_gb300 import mbe
    from paper_2607_22663_gb300.workloads import sft_problem
    prob = sft_problem([n_prompt] * batch, [n_blocks] * batch, 32, 8, 128, B, seed=7, device=dev)
    mask = mbe.sft_block_mask(prob.n_prompt_blocks, prob.n_blocks, K, prob.mask_rows)
    T, Hq, D = prob.q.shape
    Hkv = prob.k.shape[1]
    nb = n_prompt + 2 * n_blocks
    bits = mask[0].cpu().numpy().astype("int64") & 0xFFFFFFFF
    visible = sum(bin(int(w)).count("1") for w in bits[:nb].ravel())
    pairs = visible * B * B * batch
    ws = torch.empty(mbe.window_attention_workspace_size(batch, Hq, Hkv, D, prob.max_seq_len, 0), dtype=torch.uint8,
                     device=dev)
    out = torch.empty_like(prob.q)
    lse = torch.empty((T, Hq), dtype=torch.float32, device=dev)
    bws = torch.empty(int(mbe.lib().mbe_block_mask_attention_bwd_workspace_size(batch, T, Hq)), dtype=torch.uint8,
                      device=dev)
    dq = torch.empty((T, Hq, D), dtype=torch.float32, device=dev)
    dk = torch.empty((T, Hkv, D), dtype=torch.float32, device=dev)
    dv = torch.empty_like(dk)
    ms_mask = ev_time(lambda: mbe.sft_block_mask(prob.n_prompt_blocks, prob.n_blocks, K, prob.mask_rows, out=mask))
    ms_f = ev_time(lambda: mbe.block_mask_attention(prob.q, prob.k, prob.v, prob.seq_len, prob.cu_seqlens, mask,
                                                    block_size=B, max_seq_len=prob.max_seq_len, out=out, lse=lse,
                                                    workspace=ws))
    ms_b = ev_time(lambda: mbe.block_mask_attention_bwd(prob.q, prob.k, prob.v, out, prob.dout, lse, prob.seq_len,
                                                        prob.cu_seqlens, mask, block_size=B,
                                                        max_seq_len=prob.max_seq_len, dq=dq, dk=dk, dv=dv,
                                                        workspace=bws))
    tf_f = 4.0 * D * Hq * pairs / (ms_f * 1e-3) / 1e12
    tf_b = 10.0 * D * Hq * pairs / (ms_b * 1e-3) / 1e12
    return {"batch": batch, "seq_len": prob.max_seq_len, "heads_q_kv": [Hq, Hkv], "head_dim": D, "block_size": B,
            "K": K, "mask_density": round(visible / (nb * nb), 4), "mask_us": round(ms_mask * 1e3, 2),
            "fwd_ms": round(ms_f, 4), "fwd_tflops": round(tf_f, 1),
            "fwd_frac_bf16_peak_burst": round(tf_f / peaks["bf16_tflops"], 4),
            "bwd_ms": round(ms_b, 4), "bwd_tflops": round(tf_b, 1),
            "bwd_frac_bf16_peak_burst": round(tf_b / peaks["bf16_tflops"], 4),
            "note": "FLOPs of visible token pairs only; roofline bound: tensor"}


class RefreshBuffers:
    """Preallocated buffers of the targeted refresh of one pass (every layer
    reuses them; the layers run in order on one stream)."""

    def __init__(self, a0, dev, max_blocks):
        from paper_2607_22663_gb300 import mbe
        B = a0.block_size
        self.E = a0.batch * max_blocks
        self.max_prefix = max(p + B * ((wl - 1) // B) for p, wl in zip(a0.prefix_host, a0.window_host) if wl > 0)
        self.q, self.k, self.v = torch.empty_like(a0.q), torch.empty_like(a0.k_win), torch.empty_like(a0.v_win)
        self.out = torch.empty_like(a0.q)
        self.ws = torch.empty(mbe.window_attention_workspace_size(self.E, a0.num_q_heads, a0.num_kv_heads, a0.head_dim,
                                                                  B, self.max_prefix), dtype=torch.uint8, device=dev)
        self.plan = None


def refresh_pass(attn, changed, rb, stream=None):
    """Sec. 4.3 refresh of the changed blocks over every layer: plan once, then
    per layer gather the changed rows' Q/K/V, write their K/V, attend."""
    from paper_2607_22663_gb300 import mbe
    a0 = attn[0]
    B = a0.block_size
    rb.plan = mbe.refresh_plan(changed, a0.prefix_len, a0.window_len, a0.cu_window, a0.block_table, block_size=B,
                               max_window=a0.max_window, total_rows=a0.total_tokens, out=rb.plan, stream=stream)
    p = rb.plan
    for i, a in enumerate(attn):
        # the changed rows' Q/K/V compacted and their K/V written into the cache, one launch
        mbe.refresh_gather_write(a.q, a.k_win, a.v_win, p, a.k_cache, a.v_cache, out=(rb.q, rb.k, rb.v),
                                 stream=stream)
        fn = mbe.window_attention if i == 0 else mbe.window_attention_run
        fn(rb.q, rb.k, rb.v, a.k_cache, a.v_cache, p["block_table"], p["prefix_len"], p["window_len"], p["cu_window"],
           p["mask_mode"], block_size=B, max_window=B, max_prefix=rb.max_prefix, out=rb.out, workspace=rb.ws,
           stream=stream)


def time_refresh(w, dev, stream, peaks, ev_time, frac=0.125):
    """Targeted refresh of a seeded eighth of the window blocks, all layers."""
    attn = w["attn"]
    a0 = attn[0]
    B = a0.block_size
    max_blocks = (a0.max_window + B - 1) // B
    g = torch.Generator(device="cpu").manual_seed(99)
    changed = (torch.rand(a0.batch, max_blocks, generator=g) < frac).to(torch.uint8)
    nblk = [(wl + B - 1) // B for wl in a0.window_host]
    for s, n in enumerate(nblk):
        changed[s, n:] = 0
    rb = RefreshBuffers(a0, dev, max_blocks)
    d_changed = changed.to(dev)
    ms = ev_time(lambda: refresh_pass(attn, d_changed, rb))
    # algorithmic bytes of the refresh attention: each changed block reads K/V of
    # its prefix and of itself, and its Q and O
    kv_row = 2 * a0.num_kv_heads * a0.head_dim * 2
    qo_row = 2 * a0.num_q_heads * a0.head_dim * 2
    byts = 0
    for s in range(a0.batch):
        for b in range(nblk[s]):
            if changed[s, b]:
                ln = min(B, a0.window_host[s] - b * B)
                byts += (a0.prefix_host[s] + b * B + ln) * kv_row + ln * qo_row
    byts *= len(attn)
    return {"ms_per_pass": round(ms, 4), "changed_blocks": int(changed.sum()), "blocks": int(sum(nblk)),
            "layers": len(attn), "attention_gbs": round(byts / (ms * 1e-3) / 1e9, 1),
            "frac_hbm": round(byts / (ms * 1e-3) / 1e9 / peaks["hbm_gbs"], 4),
            "note": "plan + per layer (the changed rows' Q/K/V compacted and their K/V written, one launch; attention of the changed blocks)"}


def time_pass_loop(w, dev, reps=3, max_passes=5):
    """The editing loop of Sec. 4.1 (pass = window attention of every layer,
    Eq. 2 update, refresh of the changed blocks, commit) until no token
    changes or max_passes passes: one conditional-graph launch against the same
    calls issued from the host with a host read of the change count per pass."""
    from paper_2607_22663_gb300 import mbe
    from paper_2607_22663_gb300.workloads import editable_historical
    attn = w["attn"]
    ep = w["edit"]
    a0 = attn[0]
    B = a0.block_size
    R, V = ep.logits.shape
    max_blocks = (a0.max_window + B - 1) // B
    editable = editable_historical(a0.window_host, B, dev)
    outs = [torch.empty_like(a.q) for a in attn]
    ws = torch.empty(max(mbe.window_attention_workspace_size(a.batch, a.num_q_heads, a.num_kv_heads, a.head_dim,
                                                             a.max_window, a.max_prefix) for a in attn),
                     dtype=torch.uint8, device=dev)
    tokens = torch.empty_like(ep.committed)
    ident = torch.arange(R, dtype=torch.int32, device=dev)
    rb = RefreshBuffers(a0, dev, max_blocks)
    upd = mbe.denoise_update(ep.logits, ep.committed, a0.cu_window, block_size=B, mask_id=V - 1, omega_mask=0.5,
                             omega_edit=ep.tau, editable=editable, max_blocks=max_blocks)

    def one_pass(stream):
        for i, a in enumerate(attn):
            fn = mbe.window_attention if i == 0 else mbe.window_attention_run
            fn(a.q, a.k_win, a.v_win, a.k_cache, a.v_cache, a.block_table, a.prefix_len, a.window_len, a.cu_window,
               a.mask_mode, block_size=B, max_window=a.max_window, max_prefix=a.max_prefix, out=outs[i], workspace=ws,
               stream=stream)
        mbe.denoise_update(ep.logits, tokens, a0.cu_window, block_size=B, mask_id=V - 1, omega_mask=0.5,
                           omega_edit=ep.tau, editable=editable, out=upd, stream=stream)
        refresh_pass(attn, upd["block_changed"], rb, stream=stream)
        mbe.gather_rows(upd["new_tokens"], ident, out=tokens, stream=stream)

    s = torch.cuda.Stream(dev)
    with torch.cuda.stream(s):
        tokens.copy_(ep.committed)
        one_pass(s)          # allocates the refresh layout buffers outside the capture
    s.synchronize()
    passes = torch.zeros(1, dtype=torch.int32, device=dev)
    loop = mbe.PassLoop(max_passes, passes, s)
    try:
        one_pass(s)
        loop.until_stable(upd["seq_changes"])
        loop.end()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        graph_ms = []
        for r in range(reps + 1):
            with torch.cuda.stream(s):
                tokens.copy_(ep.committed)
                e0.record(s)
                loop.launch()
                e1.record(s)
            s.synchronize()
            if r:
                graph_ms.append(e0.elapsed_time(e1))
        n_graph = int(passes.item())
    finally:
        loop.close()
    eager_ms = []
    for r in range(reps + 1):
        with torch.cuda.stream(s):
            tokens.copy_(ep.committed)
            s.synchronize()
            t0 = time.perf_counter()
            n = 0
            while True:
                one_pass(s)
                n += 1
                if int(upd["seq_changes"].sum().item()) == 0 or n >= max_passes:
                    break
            s.synchronize()
            if r:
                eager_ms.append((time.perf_counter() - t0) * 1e3)
    return {"passes": n_graph, "eager_passes": n, "max_passes": max_passes,
            "graph_ms": round(statistics.median(graph_ms), 4), "eager_ms": round(statistics.median(eager_ms), 4),
            "note": "pass = window attention of every layer + Eq. 2 update + refresh of changed blocks + commit"}


def run_e2e(args, w, attention_call, edit_call, dev, stream, world, new_t, mask_t, conf_t, copy_streams=1):
    """Same pass through the public API with the per-step inputs (window Q/K/V
    of every layer, logits, committed tokens) copied from pinned host memory
    and the step's result (new tokens, edit mask, confidence) read back. The
    paged KV caches are resident state, as in serving. The copies run on
    copy_streams streams (layer l's inputs on stream l mod n, the logits in n
    slices) beside the compute stream, and layer l computes once its own inputs
    have arrived. The device input buffers are double-buffered across steps:
    step k copies into set k mod 2 as soon as step k - 2 (the last reader of that
    set) has finished, so the copies of one step overlap the compute of the one
    before and the steady state runs at max(copy time, compute time). One copy
    stream is the default: on this GPU one stream of pinned host-to-device copies
    moved about 208 GB/s, idle or beside the attention kernels, and two or four
    concurrent ones no more. Some steps' host-to-device copies stall for
    100-470 ms (seen with no kernel running as well), and the timed steps
    include whatever stalls occur."""
    attn = w["attn"]
    ep = w["edit"]
    nbuf = 2
    host = []
    dbuf = [[] for _ in range(nbuf)]
    for a in attn:
        host.append(tuple(t.cpu().pin_memory() for t in (a.q, a.k_win, a.v_win)))
        for b in range(nbuf):
            dbuf[b].append(tuple(torch.empty_like(t) for t in (a.q, a.k_win, a.v_win)))
    if ep is not None:
        lg_h = ep.logits.cpu().pin_memory()
        cm_h = ep.committed.cpu().pin_memory()
        lg_d = [torch.empty_like(ep.logits) for _ in range(nbuf)]
        cm_d = [torch.empty_like(ep.committed) for _ in range(nbuf)]
        R = ep.logits.shape[0]
        out_h = [torch.empty(R, dtype=t.dtype, pin_memory=True) for t in (new_t, mask_t, conf_t)]
        cuts = [R * k // copy_streams for k in range(copy_streams + 1)]
    cs = [torch.cuda.Stream(dev) for _ in range(copy_streams)]
    h2d = sum(t.numel() * t.element_size() for hs in host for t in hs)
    if ep is not None:
        h2d += lg_h.numel() * lg_h.element_size() + cm_h.numel() * cm_h.element_size()
    d2h = sum(t.numel() * t.element_size() for t in out_h) if ep is not None else 0
    freed = [None] * nbuf   # compute-stream event after the last read of buffer set b
    counter = [0]

    def step():
        b = counter[0] % nbuf
        counter[0] += 1
        if freed[b] is not None:
            for c in cs:
                c.wait_event(freed[b])
        copied = [torch.cuda.Event() for _ in attn]
        for i in range(len(attn)):
            with torch.cuda.stream(cs[i % copy_streams]):
                for d, h in zip(dbuf[b][i], host[i]):
                    d.copy_(h, non_blocking=True)
                copied[i].record(cs[i % copy_streams])
        done_l = []
        if ep is not None:
            for k in range(copy_streams):
                with torch.cuda.stream(cs[k]):
                    lg_d[b][cuts[k]:cuts[k + 1]].copy_(lg_h[cuts[k]:cuts[k + 1]], non_blocking=True)
                    if k == 0:
                        cm_d[b].copy_(cm_h, non_blocking=True)
                    e = torch.cuda.Event()
                    e.record(cs[k])
                    done_l.append(e)
        for i, a in enumerate(attn):
            stream.wait_event(copied[i])
            attention_call(i, a, *dbuf[b][i])
        if ep is not None:
            for e in done_l:
                stream.wait_event(e)
            edit_call(lg_d[b], cm_d[b])
            for h, d in zip(out_h, (new_t, mask_t, conf_t)):
                h.copy_(d, non_blocking=True)
        freed[b] = torch.cuda.Event()
        freed[b].record(stream)

    # warm up until two consecutive steps agree within 5% (the first large
    # copies out of freshly pinned host memory can run several times slower)
    prev = None
    for i in range(12):
        t0 = time.perf_counter()
        step()
        torch.cuda.synchronize()
        dt = time.perf_counter() - t0
        if i + 1 >= max(1, min(args.warmup, 3)) and prev is not None and abs(dt - prev) <= 0.05 * prev:
            break
        prev = dt
    K = max(1, min(args.steps, args.e2e_steps))
    if world > 1:
        torch.distributed.barrier()
    t0 = time.perf_counter()
    for _ in range(K):
        step()
    torch.cuda.synchronize()
    el = max_over_ranks(time.perf_counter() - t0, dev)
    return {"value": round(whole_job_rate(attn[0].batch * K, world, el), 3), "unit": "windows/s", "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": K, "copy_streams": copy_streams, "input_buffer_sets": nbuf,
            "h2d_gbs_effective": round(h2d * K / el / 1e9, 1),
            "resident_state": "paged KV caches of every layer (written by earlier passes)"}


# ------------------------------------------------------------------ CPU oracle arm
def run_cpu_sample(w, target_s=15.0, max_seqs=None):
    """Times the oracle on a bounded sample: a few whole sequences (all heads) of
    one layer, scaled to the workload's layer count, plus the edit decision of
    those sequences' rows. Returns windows/s and a description."""
    import numpy as np

    import oracle
    from paper_2607_22663_gb300.workloads import bf16_bits
    from paper_2607_22663_gb300.workloads import extract_sequences as subproblem

    attn = w["attn"]
    a = attn[0]
    order = np.argsort(a.prefix_host)
    # sequences near the median prefix, growing the sample until ~target_s
    mid = len(order) // 2
    picks, spent, t_attn = [], 0.0, 0.0
    rows_timed, t_edit = 0, 0.0
    ep = w["edit"]
    k = 0
    while spent < target_s and k < len(order) and (max_seqs is None or len(picks) < max_seqs):
        s = int(order[(mid + (k // 2 + 1) * (1 if k % 2 else -1)) % len(order)]) if k else int(order[mid])
        k += 1
        sub = subproblem(a, [s])
        t = time.perf_counter()
        oracle.window_attention(bf16_bits(sub.q), bf16_bits(sub.k_win), bf16_bits(sub.v_win), bf16_bits(sub.k_cache),
                                bf16_bits(sub.v_cache), sub.block_table.numpy(), sub.prefix_len.numpy(),
                                sub.window_len.numpy(), sub.cu_window.numpy(), sub.mask_mode.numpy(),
                                sub.block_size, sub.page_size)
        dt = time.perf_counter() - t
        t_attn += dt
        picks.append(s)
        spent += dt
        if ep is not None:
            t0 = int(a.cu_window[s])
            rows = list(range(t0, t0 + a.window_host[s]))
            lg = ep.logits[rows].cpu()
            t = time.perf_counter()
            if lg.dtype == torch.bfloat16:
                oracle.edit_decide(bf16_bits(lg), ep.committed[rows].cpu().numpy(), tau=ep.tau, is_bf16=True)
            else:
                oracle.edit_decide(lg.numpy(), ep.committed[rows].cpu().numpy(), tau=ep.tau)
            dt = time.perf_counter() - t
            t_edit += dt
            spent += dt
            rows_timed += len(rows)
    n = len(picks)
    per_window = t_attn / n * len(attn) + (t_edit / n if ep is not None else 0.0)
    desc = (f"{n} sequences (prefix {sorted(a.prefix_host[s] for s in picks)}), all {a.num_q_heads} heads, 1 of "
            f"{len(attn)} layers scaled x{len(attn)}; edit-decide on their {rows_timed} rows; "
            f"{spent:.1f} s of oracle time")
    return 1.0 / per_window, desc, spent


def run_reference(args, rank, world):
    import oracle
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    w = build_workload(args.workload, dev, args.layers, args.batch)
    cores = oracle.num_threads()
    # each step: one bounded sample sized so warmup+steps finish in minutes
    per_step_s = max(2.0, min(20.0, 120.0 / max(1, args.steps + args.warmup)))
    vals = []
    desc = ""
    for i in range(args.warmup + args.steps):
        v, desc, spent = run_cpu_sample(w, target_s=per_step_s)
        if i >= args.warmup:
            vals.append(v)
    value = statistics.mean(vals)
    res = {"metric": METRIC, "value": round(value, 5), "unit": "windows/s", "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": round(1000.0 / value * w["attn"][0].batch, 2) if value else None,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "impl": "reference", "config": {**workload_config(w), "parallelism": "cpu"},
           "cpu_baseline": {"value": round(value, 5), "unit": "windows/s", "cores": cores, "kind": "oracle",
                            "sample": desc},
           "e2e": {"value": round(value, 5), "unit": "windows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    return res


def run_edit_kv_case(dev, stream, peaks):
    """Edit decision over the varlen64 (4992 x 65536) and serving128 (8192 x 131072)
    logits, three calls each, then three KV window writes of one layer of the serving
    mix at 32 sequences (1.15 GB of cache, so that a multi-pass ncu capture holds a few GB
    at most); timed with CUDA events."""
    from paper_2607_22663_gb300 import mbe
    from paper_2607_22663_gb300 import workloads as wl
    res = {"profile_case": "edit_kv"}
    for rows, v in ((4992, 65536), (8192, 131072)):
        g = torch.Generator(device=dev).manual_seed(3)
        ep = wl.edit_problem(rows, v, torch.bfloat16, 3, dev, sd=2.0, peak_frac=0.6, peak_lo=2.0, peak_hi=10.0, tau=0.9,
                             g=g)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        ev[0].record(stream)
        for i in range(3):
            mbe.edit_decide(ep.logits, ep.committed, tau=ep.tau, want_argmax=False)
            ev[i + 1].record(stream)
        torch.cuda.synchronize()
        ms = statistics.median(ev[i].elapsed_time(ev[i + 1]) for i in range(3))
        gbs = edit_bytes(rows, v, 2) / (ms * 1e-3) / 1e9
        res[f"edit_decide_{rows}x{v}"] = {"ms": round(ms, 4), "gbs": round(gbs, 1),
                                          "frac_hbm": round(gbs / peaks["hbm_gbs"], 4)}
        del ep
        torch.cuda.empty_cache()
    a = build_workload("serving128", dev, 1, 32, 8)["attn"][0]
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    ev[0].record(stream)
    for i in range(3):
        mbe.kv_window_write(a.k_win, a.v_win, a.k_cache, a.v_cache, a.block_table, a.prefix_len, a.window_len,
                            a.cu_window, block_size=a.block_size, max_window=a.max_window)
        ev[i + 1].record(stream)
    torch.cuda.synchronize()
    res["kv_window_write_32_seqs_ms"] = round(statistics.median(ev[i].elapsed_time(ev[i + 1])
                                                                      for i in range(3)), 4)
    return res


def run_profile_case(args):
    """One extra on its own, for ncu captures of its kernels: the fused LM head
    (--lm-rows x 131072 x 4096 on seeded random weights, beside cuBLAS), the SFT
    attention forward and backward (--sft-seqs sequences of 4 prompt blocks and
    --sft-blocks noisy + clean blocks), edit-decide and the KV write, or the Eq. 2
    update, tail-entropy choice and targeted refresh of the serving mix (--batch,
    --layers). Three warm-up calls, then the timed ones."""
    from types import SimpleNamespace
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()
    peaks, _ = load_peaks()

    def ev_time(fn, reps=3):
        for _ in range(3):
            fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    if args.profile_case == "edit_kv":
        return run_edit_kv_case(dev, stream, peaks)
    if args.profile_case == "refresh":
        # the serving mix at --batch sequences (default 128) and --layers layers
        # (default 2): the Eq. 2 update and the tail-entropy choice over its
        # logits, then one targeted refresh pass of a seeded eighth of the blocks
        w = build_workload("serving128", dev, args.layers or 2, args.batch, args.vocab)
        res = {**time_denoise_select(w, w["attn"][0], dev, peaks, ev_time),
               "refresh": time_refresh(w, dev, stream, peaks, ev_time),
               "config": workload_config(w)}
    elif args.profile_case == "lm_head":
        R, V = args.lm_rows, 131072
        g = torch.Generator(device=dev).manual_seed(5)
        edit = SimpleNamespace(logits=torch.empty(R, V, dtype=torch.bfloat16, device=dev), tau=0.9,
                               committed=torch.randint(0, V, (R,), generator=g, device=dev, dtype=torch.int32))
        res = time_lm_head({"edit": edit}, dev, peaks, ev_time)
    elif args.profile_case == "sft":
        res = time_sft_attention(dev, peaks, ev_time, batch=args.sft_seqs, n_blocks=args.sft_blocks)
    from paper_2607_22663_gb300 import mbe
    st, flags = mbe.get_device_error()
    if st != 0:
        raise RuntimeError(f"device error: status {st} flags {flags:#x}")
    return {"profile_case": args.profile_case, **res}


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["gpu", "reference"], default="gpu")
    ap.add_argument("--workload", default="serving128",
                    choices=["serving128", "tiny", "batch8", "varlen64", "long32k"])
    ap.add_argument("--layers", type=int, default=None, help="layer count of the serving workload (default 24)")
    ap.add_argument("--batch", type=int, default=None, help="sequences of the serving workload (default 128; "
                    "smaller values are for profiling captures, not bench lines)")
    ap.add_argument("--vocab", type=int, default=None, help="vocabulary of the serving workload (default 131072; "
                    "smaller values are for profiling captures, not bench lines)")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true", help="skip the end-to-end pass and the extras (for "
                    "profiling captures; not for bench lines)")
    ap.add_argument("--profile-case", choices=["lm_head", "sft", "edit_kv", "refresh"], default=None,
                    help="time one extra on its own and print its JSON (for profiling captures; not a bench line)")
    ap.add_argument("--lm-rows", type=int, default=1024, help="rows of the --profile-case lm_head projection")
    ap.add_argument("--sft-seqs", type=int, default=4, help="sequences of the --profile-case sft batch")
    ap.add_argument("--sft-blocks", type=int, default=64, help="noisy (= clean) blocks per --profile-case sft sequence")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.profile_case is not None:
        print(json.dumps(run_profile_case(args)), flush=True)
        return

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        if rank != 0:
            return
        print(json.dumps(run_reference(args, rank, world)), flush=True)
        return
    if world > 1:
        torch.distributed.init_process_group("nccl")
    res = run_gpu(args, rank, world)
    if rank == 0:
        print(json.dumps(res), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()

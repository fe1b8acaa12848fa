"""Benchmark of the per-chunk QuantWM KV-cache path on GB300.

One step = one pass of the whole hot path for one new chunk of one layer:
  attend   -- the chunk's queries attend over the packed history (every cached
              chunk, with the PSAC logit term) and the active bf16 chunk;
  append   -- the chunk's keys/values are QSAC-assigned, INT2-quantised,
              PSAC-corrected and packed into a cache slot.
Default workload: the Wan-14B-shaped layer (40 heads, head_dim 128, chunks of
4680 tokens, 6 cached chunks = 28080 tokens, C=256, G=32, r=16, M=4).

value  = attend FLOPs of the step / step time (whole-job, all ranks), TFLOP/s;
the line also carries append GB/s and attend TFLOP/s with their roofline
fractions, an end-to-end number through the public API with host buffers,
the CPU oracle baseline and the SM clocks seen during the timed region.

--impl reference times the CPU oracle (plain C, OpenMP over heads/rows) on a
bounded sample of the same workload, scaled to the same metric.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "attend TFLOP/s + append GB/s per chunk, GB300 roofline % (1 GPU)"
UNIT = "TFLOP/s"


def workload_numbers(wl, scale_format=0):
    """Algorithmic work of one step (one layer-chunk)."""
    H, d, N, C, G, r = wl.heads, wl.head_dim, wl.chunk_tokens, wl.centroids, wl.group_size, wl.psac_rank
    L = wl.cache_tokens
    Nq = Ncur = N
    attend_flops = 2.0 * H * Nq * (L * (2 * d + r) + Ncur * 2 * d)
    ng = d // G
    scale_b = ng + 2 if scale_format else 2 * ng   # uint8 codes + binary16 secondary, or binary16 per group
    k_tok = d // 4 + scale_b + 1 + 1 + (r + 2 if r else 0)
    v_tok = d // 4 + scale_b + 1 + 1
    reads = 2 * N * H * d * 2 + 2 * H * C * d * 2 + H * d * r * 2 + H * d * 4
    writes = N * H * (k_tok + v_tok) + 2 * H * C * d * 2 + H * r * d * 2
    return {"attend_flops": attend_flops, "append_bytes": float(reads + writes),
            "append_read_bytes": float(reads), "append_write_bytes": float(writes),
            "k_bytes_per_token_head": k_tok, "v_bytes_per_token_head": v_tok}


def attend_traffic(workload):
    """DRAM bytes per attend launch from the committed ncu summary, or None when
    the kernel source has changed since those counters were taken or the
    workload is not the one they were taken on."""
    import hashlib
    prof = os.path.join(ROOT, "profiles", "attend_kernel_wan14b_layer.md")
    src = os.path.join(ROOT, "paper_2609_26425_gb300", "csrc", "attend.cu")
    try:
        fields = {}
        with open(prof) as f:
            for line in f:
                if ":" in line and line.split(":")[0] in ("traffic_bytes_per_launch", "source_sha256", "workload"):
                    k, v = line.split(":", 1)
                    fields[k.strip()] = v.strip()
        with open(src, "rb") as f:
            digest = hashlib.sha256(f.read()).hexdigest()
        if fields.get("source_sha256") == digest and fields.get("workload") == workload:
            return int(fields["traffic_bytes_per_launch"])
    except (OSError, ValueError, KeyError):
        pass
    return None


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return {"hbm_gbs": j["hbm_gbs"], "bf16_tflops": j["bf16_tflops"],
                "bf16_tflops_sustained": j.get("bf16_tflops_sustained", j["bf16_tflops"]), "src": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "src": "fallback"}


class ClockSampler:
    """nvidia-smi clock/throttle sampling during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="qwm_clocks_", suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        # the sampler is live once its first row is out; then the timed region starts
        t_end = time.time() + 5.0
        while time.time() < t_end and self.proc.poll() is None:
            if os.path.getsize(self.path) > 0:
                break
            time.sleep(0.02)

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.fh.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
                except ValueError:
                    continue
        os.unlink(self.path)
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, fl in rows for i, v in enumerate(fl) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------------------- replicas
def job_time_ms(local_ms, world, device):
    """The whole job's time: the slowest rank's (max over ranks; one rank: its own)."""
    if world <= 1:
        return float(local_ms)
    import torch
    tt = torch.tensor([float(local_ms)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(tt, op=torch.distributed.ReduceOp.MAX)
    return float(tt.item())


def whole_job_tflops(world, steps, flops_per_step, job_ms):
    """Whole-job throughput of `world` replicas, each doing `steps` steps of
    `flops_per_step` (weak scaling), over the slowest rank's time."""
    return world * steps * flops_per_step / (job_ms * 1e-3) / 1e12


# ---------------------------------------------------------------------------- GPU arm
def run_gpu(args, wl, rank, world):
    import torch
    import paper_2609_26425_gb300 as qwm
    from paper_2609_26425_gb300 import synth

    local = int(os.environ.get("LOCAL_RANK", 0))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    qwm.lib()
    H, N, C, G, r, M = wl.heads, wl.chunk_tokens, wl.centroids, wl.group_size, wl.psac_rank, wl.candidates
    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=M, kmeans_iters=wl.kmeans_iters,
                     scale_format=args.scale_format)
    src = synth.ChunkSource(wl, layer=rank)
    ws = torch.empty(qwm.qwm_fit_workspace_bytes(cfg, N), dtype=torch.uint8, device=dev)

    def chunk_inputs(t):
        q, k, v = src.chunk(t)
        a = src.query_log_scale(t)
        w = synth.population_w(a) if t > 0 else None
        U = synth.population_U(a, r) if (t > 0 and r > 0) else None
        return q, k, v, w, U

    # history: past_chunks appended through the product path (centroids fitted on the GPU)
    hist = qwm.Cache(cfg, N, wl.past_chunks, device=dev)
    past = []
    for t in range(wl.past_chunks):
        _, k, v, w, U = chunk_inputs(t)
        kd, vd = k.to(dev), v.to(dev)
        kc = qwm.qwm_fit_centroids(cfg, kd, workspace=ws)
        vc = qwm.qwm_fit_centroids(cfg, vd, workspace=ws)
        wd_t = None if w is None else w.to(dev)
        Ud_t = None if U is None else U.to(dev)
        qwm.qwm_quantize_append(cfg, hist, kd, vd, kc, vc, w=wd_t, U=Ud_t)
        past.append((kd, vd, kc, vc, wd_t, Ud_t))
    # the new chunk
    q, k, v, w, U = chunk_inputs(wl.past_chunks)
    qd, kd, vd = q.to(dev), k.to(dev), v.to(dev)
    wd = w.to(dev) if w is not None else None
    Ud = U.to(dev) if U is not None else None
    kc = qwm.qwm_fit_centroids(cfg, kd, workspace=ws)
    vc = qwm.qwm_fit_centroids(cfg, vd, workspace=ws)
    ring = qwm.Cache(cfg, N, 1, sliding_window=True, device=dev)  # the new chunk's slot
    out = torch.empty_like(qd)
    torch.cuda.synchronize()

    nums = workload_numbers(wl, args.scale_format)
    stream = torch.cuda.current_stream()
    # scratch of the balanced launch (the last wave's work units split along
    # the key chunks), allocated once outside the timed region
    aws = qwm.attend_workspace(cfg, hist, N, N, device=dev)

    def step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        qwm.qwm_attend(cfg, hist, qd, kd, vd, out=out, workspace=aws)
        if ev is not None:
            ev[1].record(stream)
        qwm.qwm_quantize_append(cfg, ring, kd, vd, kc, vc, w=wd, U=Ud)
        if ev is not None:
            ev[2].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    clocks = ClockSampler(local)
    clocks.start()
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for i in range(args.steps):
        step(evs[i])
    t1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    clk = clocks.stop()
    st = hist.status() | ring.status()
    if st:
        raise RuntimeError(f"device status {st} after the timed region")
    ms = t0.elapsed_time(t1)
    att_ms = sum(e[0].elapsed_time(e[1]) for e in evs) / args.steps
    app_ms = sum(e[1].elapsed_time(e[2]) for e in evs) / args.steps
    ms = job_time_ms(ms, world, dev)

    # ---- end to end through the public API with host buffers: every step
    # copies its inputs from pinned host memory and reads its output back; two
    # device buffer sets let the copies of one step overlap the kernels of the
    # previous one (copy-in, compute and copy-out on three streams)
    pin = lambda t: t.pin_memory()
    hq, hk, hv = pin(q), pin(k), pin(v)
    hkc, hvc = pin(kc.cpu()), pin(vc.cpu())
    hw = pin(w) if w is not None else None
    hU = pin(U) if U is not None else None
    hin = (hq, hk, hv, hkc, hvc, hw, hU)
    like = (qd, kd, vd, kc, vc, wd, Ud)
    sets = [[torch.empty_like(t) if t is not None else None for t in like] for _ in range(2)]
    outs = [torch.empty_like(qd) for _ in range(2)]
    houts = [torch.empty(out.shape, dtype=out.dtype).pin_memory() for _ in range(2)]
    h2d = sum(t.numel() * t.element_size() for t in hin if t is not None)
    d2h = houts[0].numel() * houts[0].element_size()
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev_in = [torch.cuda.Event() for _ in range(2)]
    ev_done = [torch.cuda.Event() for _ in range(2)]
    ev_out = [torch.cuda.Event() for _ in range(2)]
    for e in ev_done + ev_out:
        e.record(stream)

    def e2e_step(step):
        b = step & 1
        dq_, dk_, dv_, dkc_, dvc_, dw_, dU_ = sets[b]
        with torch.cuda.stream(s_in):
            s_in.wait_event(ev_done[b])  # the kernels that read this buffer set two steps ago are done
            for h_, d_ in zip(hin, sets[b]):
                if h_ is not None:
                    d_.copy_(h_, non_blocking=True)
            ev_in[b].record(s_in)
        stream.wait_event(ev_in[b])
        stream.wait_event(ev_out[b])  # the output buffer's previous read-back is done
        qwm.qwm_attend(cfg, hist, dq_, dk_, dv_, out=outs[b], workspace=aws)
        qwm.qwm_quantize_append(cfg, ring, dk_, dv_, dkc_, dvc_, w=dw_, U=dU_)
        ev_done[b].record(stream)
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev_done[b])
            houts[b].copy_(outs[b], non_blocking=True)
            ev_out[b].record(s_out)

    for i_ in range(max(1, args.warmup)):
        e2e_step(i_)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    s_in.wait_stream(stream)
    s_out.wait_stream(stream)
    for i_ in range(args.steps):
        e2e_step(i_)
    stream.wait_stream(s_in)
    stream.wait_stream(s_out)
    e1.record(stream)
    torch.cuda.synchronize()
    e_ms = e0.elapsed_time(e1)
    e_ms = job_time_ms(e_ms, world, dev)

    qs = query_stats_timing(qwm, cfg, qd, dev, max(3, min(args.steps, 20)), stream)
    shift = top1_shift_measure(qwm, wl, hist, past, qd, dev)
    del past
    fit_ms = fit_timing(qwm, cfg, kd, vd, ws, dev, max(3, min(args.steps, 10)), stream)

    pk = peaks()
    att_tflops = nums["attend_flops"] / (att_ms * 1e-3) / 1e12
    app_gbs = nums["append_bytes"] / (app_ms * 1e-3) / 1e9
    value = whole_job_tflops(world, args.steps, nums["attend_flops"], ms)
    e2e_value = whole_job_tflops(world, args.steps, nums["attend_flops"], e_ms)
    res = {
        "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms / args.steps, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": {"workload": wl.name, "heads": H, "head_dim": wl.head_dim, "chunk_tokens": N,
                   "cached_tokens": wl.cache_tokens, "active_tokens": N, "query_tokens": N,
                   "centroids": C, "group_size": G, "psac_rank": r, "candidates": M,
                   "scale_format": "binary16 group scales" if args.scale_format == 0 else
                   "uint8 group codes x binary16 secondary scale",
                   "parallelism": f"replicas{world}" if world > 1 else "single",
                   "l2": "inputs larger than L2 (packed history %.0f MB + q/k/v %.0f MB per step)" % (
                       hist.nbytes / 1e6, 3 * qd.numel() * 2 / 1e6)},
        # the attend kernel is timed in a sub-second region at the maximum SM
        # clock, so its roofline is the burst bf16 rate; the sustained one is
        # given beside it
        "attend": {"ms": round(att_ms, 4), "tflops": round(att_tflops, 2),
                   "frac_of_measured_bf16": round(att_tflops / pk["bf16_tflops"], 4),
                   "frac_of_measured_bf16_sustained": round(att_tflops / pk["bf16_tflops_sustained"], 4)},
        "append": {"ms": round(app_ms, 4), "gbs": round(app_gbs, 1),
                   "frac_of_measured_hbm": round(app_gbs / pk["hbm_gbs"], 4),
                   "algorithmic_bytes": nums["append_bytes"]},
        "roofline": {"bound": "tensor", "kernel": "attend_kernel", "achieved": round(att_tflops, 2),
                     "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
                     "frac": round(att_tflops / pk["bf16_tflops"], 4), "traffic": attend_traffic(None if args.scale_format else wl.name),
                     "peak_src": pk["src"] + " burst bf16 (binary16 operands run at the bf16 rate)"},
        "e2e": {"value": round(e2e_value, 3), "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        # attend: one kernel; append: the candidate filter and the quantize kernel
        # when M <= 8 and M < C, a single kernel otherwise
        "gpu_launches": (1 + (2 if (M < C and M <= 8) else 1)) * args.steps,
        "clocks": clk,
        "query_stats": {"update_ms": round(qs["update_ms"], 4),
                        "update_gbs": round(qs["update_bytes"] / (qs["update_ms"] * 1e-3) / 1e9, 1),
                        "update_frac_of_measured_hbm": round(
                            qs["update_bytes"] / (qs["update_ms"] * 1e-3) / 1e9 / pk["hbm_gbs"], 4),
                        "update_algorithmic_bytes": qs["update_bytes"],
                        "basis_ms": round(qs["basis_ms"], 4), "jacobi_sweeps": qs["sweeps"],
                        "l2": "update: 4 rotating copies of q (192 MB); basis: 256 MB flush before each launch"},
        # quality: share of queries whose highest-logit cached key moves away from the bf16 keys' one
        "top1_shift": shift,
        # chunk boundary, not on the step: Lloyd k-means tables of the chunk's Keys and Values
        "fit": {"ms_keys_and_values": round(fit_ms, 3), "kmeans_iters": wl.kmeans_iters,
                "l2": "256 MB flush before each timed pair"},
    }
    return res


def top1_shift_measure(qwm, wl, hist, past, qd, dev, every=9):
    """Token-selection shift on the layer: the new chunk's queries (every 9th)
    against the cached keys reconstructed from three caches of the same past
    chunks: QVG (w = 1, nearest centroid, no PSAC), QSAC (w, top-M) and the
    bench's own QSAC + PSAC cache; the reference is the bf16 keys."""
    import torch
    H, N, C, G, r, M = wl.heads, wl.chunk_tokens, wl.centroids, wl.group_size, wl.psac_rank, wl.candidates
    qs = qd[::every].contiguous()
    sf = hist.cfg.scale_format
    cfg_ref = qwm.config(H, C, group_size=G, psac_rank=r, candidates=M, scale_format=sf)
    k_ref = torch.cat([p[0].float() for p in past])
    idx_ref = qwm.qwm_top1_keys(cfg_ref, qs, k_ref)
    del k_ref
    out = {}
    variants = (("qvg", qwm.config(H, C, group_size=G, psac_rank=0, candidates=1, scale_format=sf), False, False),
                ("qsac", qwm.config(H, C, group_size=G, psac_rank=0, candidates=M, scale_format=sf), True, False),
                ("qsac_psac", cfg_ref, True, True))
    for name, cfg, use_w, use_U in variants:
        if name == "qsac_psac":
            cache = hist
        else:
            cache = qwm.Cache(cfg, N, wl.past_chunks, device=dev)
            for kd, vd, kc, vc, w, U in past:
                qwm.qwm_quantize_append(cfg, cache, kd, vd, kc, vc, w=w if use_w else None, U=U if use_U else None)
        k_hat = torch.cat([qwm.qwm_dequant_chunk(cfg, cache, i)[0] for i in range(cache.num_chunks)])
        idx = qwm.qwm_top1_keys(cfg, qs, k_hat)
        out[name] = round(float((idx != idx_ref).float().mean().item()), 4)
        if cache.status():
            raise RuntimeError(f"device status after the {name} cache")
        del k_hat
    out["queries"] = f"{qs.shape[0]} of {qd.shape[0]} (every {every}th) x {H} heads"
    out["keys"] = int(sum(p[0].shape[0] for p in past))
    out["reference"] = "bf16 keys, fp32 channel-order logits"
    return out


def fit_timing(qwm, cfg, kd, vd, ws, dev, iters, stream):
    """qwm_fit_centroids on the chunk's Keys and then its Values (the two
    tables a chunk boundary fits), timed with CUDA events after an L2 flush."""
    import torch
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    kc = qwm.qwm_fit_centroids(cfg, kd, workspace=ws)
    vc = qwm.qwm_fit_centroids(cfg, vd, workspace=ws)
    ms = []
    for _ in range(iters):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        qwm.qwm_fit_centroids(cfg, kd, centroids=kc, workspace=ws)
        qwm.qwm_fit_centroids(cfg, vd, centroids=vc, workspace=ws)
        e1.record(stream)
        torch.cuda.synchronize()
        ms.append(e0.elapsed_time(e1))
    return sum(ms) / len(ms)


def query_stats_timing(qwm, cfg, qd, dev, iters, stream):
    """Chunk-boundary Query statistics: qwm_query_stats_update over the chunk's
    Queries (back to back over inputs larger than L2) and qwm_query_basis (w and
    U_r, each launch timed alone after an L2 flush), with CUDA events."""
    import torch
    st = qwm.QueryStats(cfg, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for _ in range(3):
        st.update(qd)
        st.basis()

    def timed(fn):
        ms = []
        for _ in range(iters):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            torch.cuda.synchronize()
            ms.append(e0.elapsed_time(e1))
        return sum(ms) / len(ms)

    # back-to-back updates over four copies of the chunk's Queries (192 MB
    # together, more than L2), one event pair around the batch
    qbufs = [qd.clone() for _ in range(4)]
    flush.zero_()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(4 * iters):
        st.update(qbufs[i % 4])
    e1.record(stream)
    torch.cuda.synchronize()
    upd = e0.elapsed_time(e1) / (4 * iters)
    del qbufs
    bas = timed(lambda: st.basis())
    status, _ = st.read()
    if status:
        raise RuntimeError(f"query statistics device status {status}")
    H, d = cfg.num_heads, cfg.head_dim
    nbytes = qd.numel() * qd.element_size() + 2 * H * d * d * 4
    return {"update_ms": upd, "basis_ms": bas, "update_bytes": nbytes, "sweeps": st.sweeps()}


# ---------------------------------------------------------------------------- layer stacks
def stack_flops(wl, r, cached_tokens):
    """Attend FLOPs of one chunk step over every layer of a stack."""
    H, N, d = wl.heads, wl.chunk_tokens, wl.head_dim
    return wl.layers * 2.0 * H * N * (cached_tokens * (2 * d + r) + N * 2 * d)


def run_stack(args, wl, psac_rank=None, distinct_layers=4):
    """Per-chunk time of a stack of layers: at every chunk step, each layer's
    new chunk attends its cached chunks and itself (bf16), then is appended;
    the step's times are summed over the layers (CUDA events around each
    call), with the packed bytes the caches hold against bf16 K/V of the same
    tokens.  Layer l draws the seeded inputs of layer l mod distinct_layers
    (the timing does not depend on the draw; drawing every layer's inputs on
    the host would take minutes).  Centroid tables: the GPU k-means of each
    chunk (10 Lloyd iterations)."""
    import torch
    import paper_2609_26425_gb300 as qwm
    from paper_2609_26425_gb300 import synth
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    qwm.lib()
    r = wl.psac_rank if psac_rank is None else psac_rank
    H, N, C, G, M, d = wl.heads, wl.chunk_tokens, wl.centroids, wl.group_size, wl.candidates, wl.head_dim
    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=M, kmeans_iters=wl.kmeans_iters,
                     scale_format=args.scale_format)
    # without a window the last step attends past_chunks chunks and then
    # appends one more; a window wraps around for two more steps at the end
    slots = wl.window if wl.window else wl.past_chunks + 1
    n_chunks = wl.past_chunks + (3 if wl.window else 1)
    Dl = min(distinct_layers, wl.layers)
    ws = torch.empty(qwm.qwm_fit_workspace_bytes(cfg, N), dtype=torch.uint8, device=dev)
    data = []
    for layer in range(Dl):
        src = synth.ChunkSource(wl, layer=layer)
        row = []
        for t in range(n_chunks):
            q, k, v = src.chunk(t)
            a = src.query_log_scale(t)
            qd, kd, vd = q.to(dev), k.to(dev), v.to(dev)
            kc = qwm.qwm_fit_centroids(cfg, kd, workspace=ws)
            vc = qwm.qwm_fit_centroids(cfg, vd, workspace=ws)
            w = synth.population_w(a).to(dev) if t > 0 else None
            U = synth.population_U(a, r).to(dev) if (t > 0 and r > 0) else None
            row.append((qd, kd, vd, kc, vc, w, U))
        data.append(row)
    caches = [qwm.Cache(cfg, N, slots, sliding_window=bool(wl.window), device=dev) for _ in range(wl.layers)]
    stream = torch.cuda.current_stream()
    out = torch.empty(N, H, d, dtype=torch.bfloat16, device=dev)
    for layer in range(wl.layers):   # chunk 0, cold start (w = 1, no PSAC): append only
        _, kd, vd, kc, vc, w, U = data[layer % Dl][0]
        qwm.qwm_quantize_append(cfg, caches[layer], kd, vd, kc, vc, w=w, U=U)
    # scratch for the balanced launch, sized for the largest cache of the run
    aws = torch.empty(max(qwm.qwm_attend_workspace_bytes(cfg, caches[0], N, N), 1) + 256, dtype=torch.uint8,
                      device=dev)
    aws = aws[(-aws.data_ptr()) % 256:]
    for _ in range(3):                # warm-up of the attention path
        qwm.qwm_attend(cfg, caches[0], data[0][1][0], data[0][1][1], data[0][1][2], out=out)
    torch.cuda.synchronize()
    lay = caches[0].layout()
    clocks = ClockSampler(0)
    clocks.start()
    rows = []
    for t in range(1, n_chunks):
        cached = caches[0].num_chunks
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(wl.layers)]
        for layer in range(wl.layers):
            qd, kd, vd, kc, vc, w, U = data[layer % Dl][t]
            need = qwm.qwm_attend_workspace_bytes(cfg, caches[layer], N, N)
            if need > aws.numel():
                aws = torch.empty(need + 256, dtype=torch.uint8, device=dev)
                aws = aws[(-aws.data_ptr()) % 256:]
            evs[layer][0].record(stream)
            qwm.qwm_attend(cfg, caches[layer], qd, kd, vd, out=out, workspace=aws if need else None)
            evs[layer][1].record(stream)
            qwm.qwm_quantize_append(cfg, caches[layer], kd, vd, kc, vc, w=w, U=U)
            evs[layer][2].record(stream)
        torch.cuda.synchronize()
        att = sum(e[0].elapsed_time(e[1]) for e in evs)
        app = sum(e[1].elapsed_time(e[2]) for e in evs)
        held = caches[0].num_chunks
        flops = stack_flops(wl, r, cached * N)
        nums = workload_numbers(wl, args.scale_format)
        rows.append({"step": t, "cached_tokens": cached * N, "attend_ms": round(att, 3), "append_ms": round(app, 3),
                     "attend_tflops": round(flops / (att * 1e-3) / 1e12, 1),
                     "append_gbs": round(wl.layers * nums["append_bytes"] / (app * 1e-3) / 1e9, 1),
                     "cache_gib": round(wl.layers * (lay.header_bytes + held * lay.slot_bytes) / 2**30, 3),
                     "bf16_gib": round(wl.layers * held * N * H * d * 2 * 2 / 2**30, 3)})
    clk = clocks.stop()
    for c in caches:
        if c.status():
            raise RuntimeError("device status after the stack run")
    return rows, clk, r


def stack_line(args, wl, psac_rank=None):
    rows, clk, r = run_stack(args, wl, psac_rank)
    pk = peaks()
    # a window: the steps with the window full; no window: the last step
    full = [x for x in rows if x["cached_tokens"] == wl.window * wl.chunk_tokens] if wl.window else rows[-1:]
    last = full[-1] if full else rows[-1]
    att_ms = sum(x["attend_ms"] for x in full) / len(full)
    app_ms = sum(x["append_ms"] for x in full) / len(full)
    flops = stack_flops(wl, r, last["cached_tokens"])
    tflops = flops / (att_ms * 1e-3) / 1e12
    nums = workload_numbers(wl, args.scale_format)
    res = {
        "metric": METRIC, "value": round(tflops, 3), "unit": UNIT, "n_gpus": 1, "steps": len(rows), "warmup": 3,
        "ms_per_step": round(att_ms + app_ms, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": {"workload": wl.name, "layers": wl.layers, "heads": wl.heads, "chunk_tokens": wl.chunk_tokens,
                   "cache_chunks": wl.window or wl.past_chunks, "sliding_window": bool(wl.window),
                   "centroids": wl.centroids, "group_size": wl.group_size, "psac_rank": r,
                   "candidates": wl.candidates, "inputs": "4 seeded layers cycled over the stack",
                   "value": ("mean over the steps with a full window" if wl.window else "the last step (the full cache)") +
                            ": attend FLOPs of all layers / summed attend time"},
        "attend": {"ms": round(att_ms, 3), "tflops": round(tflops, 2),
                   "frac_of_measured_bf16": round(tflops / pk["bf16_tflops"], 4)},
        "append": {"ms": round(app_ms, 3),
                   "gbs": round(wl.layers * nums["append_bytes"] / (app_ms * 1e-3) / 1e9, 1),
                   "frac_of_measured_hbm": round(wl.layers * nums["append_bytes"] / (app_ms * 1e-3) / 1e9 /
                                                 pk["hbm_gbs"], 4)},
        "roofline": {"bound": "tensor", "kernel": "attend_kernel", "achieved": round(tflops, 2),
                     "peak": pk["bf16_tflops"], "unit": "TFLOP/s", "frac": round(tflops / pk["bf16_tflops"], 4),
                     "traffic": None, "peak_src": pk["src"] + " burst bf16"},
        "gpu_launches": (1 + 2) * wl.layers * len(rows),
        "clocks": clk, "per_step": rows,
    }
    if not args.no_cpu_baseline:
        cb = cpu_baseline(wl, args.cpu_threads, f=0.25, f_single=0.02)
        cb["note"] = "one layer's step sampled (every layer does the same work per FLOP)"
        res["cpu_baseline"] = cb
    return res


# ---------------------------------------------------------------------------- microbench sweep
def run_sweep(args, Ns=(1024, 4096, 16384, 65536), Ls=(4096, 16384, 65536, 131072), Cs=(16, 64, 256),
              rs=(0, 8, 16, 32), Gs=(32, 64), H=40, reps=3):
    """The one-layer microbench sweep (40 heads): attend over every N x L x r
    (C = 256, G = 32; N_q = N_cur = N; caches built from 4096-token chunks),
    and quantize-append over every N x C x r x G (k-means tables of the chunk,
    10 Lloyd iterations); each point timed with CUDA events after an L2
    flush, as throughput and fraction of the measured roofline."""
    import torch
    import paper_2609_26425_gb300 as qwm
    from paper_2609_26425_gb300 import synth
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    qwm.lib()
    pk = peaks()
    d = 128
    wl = synth.Workload("sweep", heads=H, chunk_tokens=max(Ns), past_chunks=0, centroids=256, group_size=32,
                        psac_rank=16, seed=4)
    src = synth.ChunkSource(wl)
    q, k, v = src.chunk(0)
    a = src.query_log_scale(0)
    qd, kd, vd = q.to(dev), k.to(dev), v.to(dev)
    w = synth.population_w(a).to(dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def timed(fn):
        fn()
        torch.cuda.synchronize()
        ms = []
        for _ in range(reps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            torch.cuda.synchronize()
            ms.append(e0.elapsed_time(e1))
        return sorted(ms)[len(ms) // 2]

    attend_pts = []
    Lc = 4096
    for r in rs:
        cfg = qwm.config(H, 256, group_size=32, psac_rank=r, candidates=4)
        U = synth.population_U(a, r).to(dev) if r > 0 else None
        cache = qwm.Cache(cfg, Lc, max(Ls) // Lc, device=dev)
        kc = kd[: 256 * (Lc // 256): Lc // 256].transpose(0, 1).contiguous()   # strided tokens as tables
        vc = vd[: 256 * (Lc // 256): Lc // 256].transpose(0, 1).contiguous()
        for i in range(max(Ls) // Lc):
            o = (i % (max(Ns) // Lc)) * Lc
            qwm.qwm_quantize_append(cfg, cache, kd[o:o + Lc], vd[o:o + Lc], kc, vc, w=w, U=U)
            L = (i + 1) * Lc
            if L in Ls:
                for N in Ns:
                    out = torch.empty(N, H, d, dtype=torch.bfloat16, device=dev)
                    aws = qwm.attend_workspace(cfg, cache, N, N, device=dev)
                    ms = timed(lambda: qwm.qwm_attend(cfg, cache, qd[:N], kd[:N], vd[:N], out=out, workspace=aws))
                    fl = 2.0 * H * N * (L * (2 * d + r) + N * 2 * d)
                    tf = fl / (ms * 1e-3) / 1e12
                    attend_pts.append({"N": N, "L": L, "r": r, "ms": round(ms, 4), "tflops": round(tf, 1),
                                       "frac_bf16": round(tf / pk["bf16_tflops"], 4)})
        if cache.status():
            raise RuntimeError("device status after the attend sweep")
        del cache
    append_pts = []
    for N in Ns:
        kN, vN = kd[:N].contiguous(), vd[:N].contiguous()
        for C in Cs:
            cfit = qwm.config(H, C, kmeans_iters=10)
            kc = qwm.qwm_fit_centroids(cfit, kN)
            vc = qwm.qwm_fit_centroids(cfit, vN)
            for r in rs:
                U = synth.population_U(a, r).to(dev) if r > 0 else None
                for G in Gs:
                    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=4)
                    ring = qwm.Cache(cfg, N, 1, sliding_window=True, device=dev)
                    ms = timed(lambda: qwm.qwm_quantize_append(cfg, ring, kN, vN, kc, vc, w=w, U=U))
                    if ring.status():
                        raise RuntimeError("device status after an append point")
                    wlp = synth.Workload("p", heads=H, chunk_tokens=N, past_chunks=0, centroids=C, group_size=G,
                                         psac_rank=r)
                    nb = workload_numbers(wlp)["append_bytes"]
                    gbs = nb / (ms * 1e-3) / 1e9
                    append_pts.append({"N": N, "C": C, "r": r, "G": G, "ms": round(ms, 4), "gbs": round(gbs, 1),
                                       "frac_hbm": round(gbs / pk["hbm_gbs"], 4)})
                    del ring
    return {"metric": "one-layer microbench sweep (40 heads): attend TFLOP/s and append GB/s per point",
            "unit": "TFLOP/s | GB/s", "data": "synthetic", "dtype": "f16",
            "peaks": {"bf16_tflops": pk["bf16_tflops"], "hbm_gbs": pk["hbm_gbs"], "src": pk["src"]},
            "attend": attend_pts, "append": append_pts,
            "l2": "256 MB flush before each timed call; median of %d" % reps}


# ---------------------------------------------------------------------------- CPU oracle
def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the machine type)."""
    import platform
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return platform.machine()


class OracleStep:
    """The CPU oracle on a bounded sample of one step of a workload.

    A sample of fraction f holds round(f N) appended tokens (Keys and Values,
    every head), round(f 2048) query rows of 8 heads attending over every key,
    and the reconstruction of the sampled tokens; its time is measured, and the
    time of a whole step is extrapolated from it by the ratio of the work.
    Inputs are built once and are not part of the time."""

    ATT_HEADS = 8

    def __init__(self, wl):
        import numpy as np
        from oracle import oracle as orc
        from paper_2609_26425_gb300 import synth
        self.wl, self.orc, self.np = wl, orc, np
        H, N, C, r = wl.heads, wl.chunk_tokens, wl.centroids, wl.psac_rank
        src = synth.ChunkSource(wl)
        q, k, v = src.chunk(wl.past_chunks)
        self.kb, self.vb, self.qb = synth.bits(k), synth.bits(v), synth.bits(q)
        a = src.query_log_scale(wl.past_chunks)
        self.w = synth.population_w(a).numpy()
        self.Ub = synth.bits(synth.population_U(a, r))
        idx = (np.arange(C) * N) // C
        self.kc = np.ascontiguousarray(self.kb[idx].transpose(1, 0, 2))
        self.vc = np.ascontiguousarray(self.vb[idx].transpose(1, 0, 2))
        self.hs = list(range(min(self.ATT_HEADS, H)))
        self.L = wl.cache_tokens + N
        rng = np.random.default_rng(0)
        self.Kf = rng.standard_normal((self.L, len(self.hs), wl.head_dim))
        self.Vf = rng.standard_normal((self.L, len(self.hs), wl.head_dim))
        self.qs = np.ascontiguousarray(self.qb[:, self.hs])

    def run(self, f, nthreads):
        """Run a sample of fraction f; returns (measured seconds, extrapolated
        seconds of a whole step, description)."""
        wl, orc, np = self.wl, self.orc, self.np
        H, N, G, r, M = wl.heads, wl.chunk_tokens, wl.group_size, wl.psac_rank, wl.candidates
        n_app = max(16, min(N, int(round(f * N))))
        rows_n = max(4, min(N, int(round(f * 2048))))
        nh = len(self.hs)
        t0 = time.perf_counter()
        ko = orc.quantize(self.kb[:n_app], self.kc, G=G, r=r, M=M, is_key=True, w=self.w, U_bits=self.Ub,
                          nthreads=nthreads)
        orc.quantize(self.vb[:n_app], self.vc, G=G, r=r, M=M, is_key=False, nthreads=nthreads)
        t1 = time.perf_counter()
        sub = {kk: vv[:, self.hs] for kk, vv in ko.items() if isinstance(vv, np.ndarray) and vv.ndim >= 2}
        orc.dequant(sub, self.kc[self.hs], G=G, r=r, U_bits=self.Ub[self.hs])
        t2 = time.perf_counter()
        orc.attend(self.qs, self.Kf, self.Vf, 1 / math.sqrt(wl.head_dim),
                   rows=np.arange(rows_n, dtype=np.int64), nthreads=nthreads)
        t3 = time.perf_counter()
        t_app, t_deq, t_att = t1 - t0, t2 - t1, t3 - t2
        full = (t_app * N / n_app + t_deq / (n_app * nh) * 2 * wl.cache_tokens * H
                + t_att * (N / rows_n) * (H / nh))
        desc = (f"append: {n_app} of {N} tokens x {H} heads (K+V), scaled x{N / n_app:.1f}; attend: {rows_n} "
                f"query rows x {nh} of {H} heads over all {self.L} keys, scaled x{(N / rows_n) * (H / nh):.0f}; "
                f"reconstruction of {n_app} tokens x {nh} heads, scaled to the {wl.cache_tokens}-token cache")
        return t3 - t0, full, desc


def cpu_baseline(wl, nthreads, f=1.0, f_single=0.05):
    """The oracle on a bounded sample of the bench's step (all host cores, and
    once on one core), as a reported baseline."""
    from oracle import oracle as orc
    cores = nthreads if nthreads > 0 else orc.max_threads()
    ostep = OracleStep(wl)
    spent, full, desc = ostep.run(f, nthreads)
    spent1, full1, desc1 = ostep.run(f_single, 1)
    nums = workload_numbers(wl)
    return {"value": round(nums["attend_flops"] / full / 1e12, 6), "unit": UNIT, "cores": cores,
            "kind": "oracle", "cpu": cpu_model(), "sample": desc, "sample_seconds": round(spent, 2),
            "seconds_per_step_extrapolated": round(full, 2),
            "single_thread": {"value": round(nums["attend_flops"] / full1 / 1e12, 6), "sample": desc1,
                              "sample_seconds": round(spent1, 2), "seconds_per_step_extrapolated": round(full1, 2)}}


def run_reference(args, wl, budget_s=150.0):
    """The reference arm: the CPU oracle, as it stands, on the host cores.
    Each step is a bounded sample of the workload's step (OracleStep), sized
    so that warm-up and timed steps together take about budget_s seconds;
    ms_per_step is the sample's measured time and the value is the metric of
    the whole step extrapolated from it."""
    from oracle import oracle as orc
    orc.build()
    nthreads = args.cpu_threads
    cores = nthreads if nthreads > 0 else orc.max_threads()
    ostep = OracleStep(wl)
    f0 = 0.01
    t_cal, _, _ = ostep.run(f0, nthreads)          # calibration, the first warm-up step
    per_step = min(10.0, budget_s / (args.steps + args.warmup))
    f = max(f0, min(1.0, f0 * per_step / max(t_cal, 1e-3)))
    for _ in range(args.warmup - 1):
        ostep.run(f, nthreads)
    spent, fulls, desc = [], [], ""
    for _ in range(args.steps):
        t, full, desc = ostep.run(f, nthreads)
        spent.append(t)
        fulls.append(full)
    nums = workload_numbers(wl, args.scale_format)
    sec = sum(fulls) / len(fulls)
    value = nums["attend_flops"] / sec / 1e12
    ms = 1e3 * sum(spent) / len(spent)
    return {"metric": METRIC, "value": round(value, 6), "unit": UNIT, "impl": "reference", "n_gpus": 0,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 1),
            "ms_per_step_note": "measured time of one bounded sample (the step); the value is extrapolated "
                                "from it to the whole step's work",
            "ms_per_full_step_extrapolated": round(sec * 1e3, 1),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32/f64",
            "data": "synthetic", "config": {"workload": wl.name, "heads": wl.heads, "chunk_tokens": wl.chunk_tokens,
                                            "cached_tokens": wl.cache_tokens},
            "cpu_baseline": {"value": round(value, 6), "unit": UNIT, "cores": cores, "kind": "oracle",
                             "cpu": cpu_model(), "sample": desc, "sample_fraction": round(f, 4)},
            "e2e": {"value": round(value, 6), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=40)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="qwm", choices=["qwm", "reference"])
    ap.add_argument("--workload", default="wan14b_layer")
    ap.add_argument("--cpu-threads", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--scale-format", type=int, default=0, choices=[0, 1],
                    help="group scale storage: 0 binary16 per group, 1 uint8 codes + binary16 per token")
    ap.add_argument("--heads", type=int, default=0,
                    help="profiling only: the workload with fewer heads (same per-head work); not a bench line")
    ap.add_argument("--psac-rank", type=int, default=-1,
                    help="layer stacks: PSAC rank other than the workload's own (the 1.3B DiT at r = 32)")
    ap.add_argument("--sweep", action="store_true",
                    help="the one-layer microbench sweep (N x L x C x r x G); prints one JSON object")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    from paper_2609_26425_gb300 import synth
    wl = synth.WORKLOADS[args.workload]
    if args.heads > 0:
        import dataclasses
        wl = dataclasses.replace(wl, heads=args.heads, name=f"{wl.name}_h{args.heads}")
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))

    if args.sweep and args.impl != "reference":
        print(json.dumps(run_sweep(args)), flush=True)
        return
    if wl.layers > 1 and args.impl != "reference":
        print(json.dumps(stack_line(args, wl, None if args.psac_rank < 0 else args.psac_rank)), flush=True)
        return

    if args.impl == "reference":
        if rank != 0:
            return
        print(json.dumps(run_reference(args, wl)), flush=True)
        return

    if world > 1:
        import torch
        torch.distributed.init_process_group("nccl")
    res = run_gpu(args, wl, rank, world)
    if world > 1:
        import torch
        torch.distributed.destroy_process_group()
    if rank == 0:
        if not args.no_cpu_baseline and world == 1:
            res["cpu_baseline"] = cpu_baseline(wl, args.cpu_threads)
        print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()

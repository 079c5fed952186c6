#!/usr/bin/env python
"""Benchmark of the HeadGuard mixed-precision KV-cache path on one GB300.

One step = the whole path over one synthetic cache: quantize-pack every layer
from its BF16 prefill (one launch per 64 layers), then `decode_steps` decode
steps, each appending one token per (layer, row, KV head) and running decode
attention over all layers (one launch each).  Inputs are resident in HBM when
timing starts; L2 is flushed (a 512 MiB write, then a read of it so the
evicted lines are clean) before every timed launch group, and every group is
timed with CUDA events on the launching stream.

value     = algorithmic bytes of a step / summed device time of the step (GB/s)
roofline  = decode attention (the dominant kernel): its algorithmic bytes per
            launch / its mean event-timed duration, against MEASURED_PEAKS.json
e2e       = the same bytes / time of a step driven from pinned HOST buffers
            through the C ABI (H2D of prefill, queries and new K/V; D2H of
            the attention outputs inside the timed region)
--impl reference times the CPU oracle on a bounded sample of the same step.
"""
import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = ("decode-attn + quantize achieved HBM GB/s (% of 8 TB/s) and decode tokens/s, 1 GB300")
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
L2_FLUSH_BYTES = 512 << 20


def parse_args():
    return parse_args_from(None)


def parse_args_from(argv):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="headguard", choices=["headguard", "reference"])
    ap.add_argument("--workload", default="qwen25vl7b")
    ap.add_argument("--meta-bits", type=int, default=64, choices=[64, 32],
                    help="metadata per group: fp32 pair (64) or binary16 pair (32, Sec. 5.4)")
    ap.add_argument("--bits", type=int, default=0, choices=[0, 2, 3, 4],
                    help="code width override (0: the workload's own)")
    ap.add_argument("--layers", type=int, default=0,
                    help="layer-count override (0: the workload's own), e.g. for a small profile")
    ap.add_argument("--salient-permille", type=int, default=0,
                    help="AKVQ-style salient tokens kept BF16 per head (Sec. 4; 20 = 2%%)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-variants", action="store_true",
                    help="skip the per-layer-launch and graph-replay decode variants")
    return ap.parse_args(argv)


# ---------------------------------------------------------------------------
# Algorithmic bytes (inputs read + outputs written, no workspace traffic)
# ---------------------------------------------------------------------------

def geometry_bytes(runner):
    """Algorithmic bytes of quantize (per step), decode (per decode step, list),
    append (per decode step), from the library's region map."""
    import paper_2609_35800_gb300 as hg
    w = runner.w
    B, H, T = w.batch, w.kv_heads, w.seq_len
    code_tok = 128 * w.bits // 8
    q_rows = w.layers * B * w.q_heads * 256
    quant = 0
    dec_static = 0          # cache bytes read per decode step excluding appended tokens
    bf16_heads = 0          # (layer, head) pairs: appended tokens are read per head
    for l in range(w.layers):
        for h in range(H):
            r = hg.hg_cache_head_regions(runner.cache, l, h)
            nq = r.n_coded  # coded tokens (image tokens less any salient ones)
            per_b_write = r.bf16_prefill * 512
            per_b_read_dec = r.bf16_prefill * 512
            if r.head_class == hg.HG_HEAD_QUANTIZED:
                per_b_write += r.sal_bstride  # salient-token map (zero without salient tokens)
                per_b_write += nq * code_tok + r.kqm_bstride + nq * code_tok + r.vqm_bstride
                per_b_read_dec += nq * code_tok + r.kqm_bstride + nq * code_tok + r.vqm_bstride
            elif r.head_class == hg.HG_HEAD_KEYS_ONLY:
                per_b_write += r.sal_bstride
                per_b_write += nq * 256 + nq * code_tok + r.vqm_bstride
                per_b_read_dec += nq * 256 + nq * code_tok + r.vqm_bstride
            quant += B * (T * 512 + per_b_write)
            dec_static += B * per_b_read_dec
            bf16_heads += 1
    decode = []
    for s in range(w.decode_steps):
        appended = s + 1
        decode.append(dec_static + bf16_heads * B * appended * 512 + 2 * q_rows)
    append = 4 * w.layers * B * H * 256
    return quant, decode, append


# ---------------------------------------------------------------------------
# clocks
# ---------------------------------------------------------------------------

CLOCK_FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons around a timed
    region: entering waits (up to `start_timeout` s) for the first sample so
    the sampler is live when the region starts; `summary` keeps the samples
    that arrived inside the region (plus the first one after it, which covers
    its tail), or every sample when none did."""

    def __init__(self, device_index, period_ms=50, start_timeout=5.0, cmd=None):
        self.proc = None
        self.idx = device_index
        self.period_ms = period_ms
        self.start_timeout = start_timeout
        self.cmd = cmd or ["nvidia-smi"]
        self.stamped = []
        self.lines = []
        self.t0 = self.t1 = None
        self._reader = None

    def _read(self):
        for line in self.proc.stdout:
            if line.strip():
                self.stamped.append((time.perf_counter(), line))

    def __enter__(self):
        import threading
        try:
            self.proc = subprocess.Popen(
                self.cmd + ["--query-gpu=" + CLOCK_FIELDS, "--format=csv,noheader,nounits",
                            "-i", str(self.idx), "-lms", str(self.period_ms)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        if self.proc is not None:
            self._reader = threading.Thread(target=self._read, daemon=True)
            self._reader.start()
            deadline = time.perf_counter() + self.start_timeout
            while not self.stamped and self.proc.poll() is None and time.perf_counter() < deadline:
                time.sleep(0.01)
        self.t0 = time.perf_counter()
        return self

    def __exit__(self, *exc):
        self.t1 = time.perf_counter()
        if self.proc is not None:
            # let the sample in progress at the region's end arrive
            deadline = self.t1 + 2.5 * self.period_ms * 1e-3
            while (self.proc.poll() is None and time.perf_counter() < deadline
                   and not any(t >= self.t1 for t, _ in self.stamped)):
                time.sleep(0.01)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.proc.wait()
            self._reader.join(timeout=5)
        inside = [l for t, l in self.stamped if self.t0 <= t < self.t1]
        after = [l for t, l in self.stamped if t >= self.t1][:1]
        self.lines = (inside + after) or [l for _, l in self.stamped]

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in getattr(self, "lines", []):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# roofline inputs
# ---------------------------------------------------------------------------

def max_over_ranks(value, dist, device):
    """The slowest rank's value (the timing rule for N > 1 ranks: max over
    ranks after a barrier); `dist` is torch.distributed or None for one rank."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_gbs(world, step_bytes, ms_step):
    """Whole-job throughput: every rank streams its own replica's step bytes
    (weak scaling; the path has no cross-rank exchange) in the slowest rank's
    time."""
    return world * step_bytes / (ms_step * 1e-3) / 1e9


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return json.load(f), "measured"
    except (OSError, ValueError):
        return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


# the sources the decode kernel and its launch plan are built from
DECODE_SOURCES = ("hg_api.cu", "hg_common.cuh", "hg_decode.cu", "hg_decode_kernel.cuh", "hg_decode_m16.cu",
                  "hg_internal.h", "hg_layout.cuh", "hg_mma.cuh")


def kernel_source_hash():
    """Hash of the decode kernel's sources (the ncu traffic figure is valid
    while they are unchanged)."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_35800_gb300", "csrc")
    for name in DECODE_SOURCES:
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + f.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload):
    """DRAM bytes per decode launch from the committed ncu summary, if it was
    taken on the current kernel sources (else None)."""
    path = os.path.join(ROOT, "profiles", "decode_attention_%s.md" % workload)
    try:
        txt = open(path).read()
    except OSError:
        return None
    m_src = re.search(r"source_sha256_16:\s*([0-9a-f]+)", txt)
    m_tr = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", txt)
    if not m_src or not m_tr or m_src.group(1) != kernel_source_hash():
        return None
    return float(m_tr.group(1))


# ---------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline and the reference arm)
# ---------------------------------------------------------------------------

def cpu_model():
    """Host CPU model string (lscpu, else /proc/cpuinfo, else the machine type)."""
    import platform
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return platform.machine()


def oracle_sample(w, n_layers, n_steps, parts=None):
    """Time the oracle on the first n_layers layers: quantize, then n_steps decode
    steps of attention over those layers.  Returns (bytes, seconds, threads);
    with `parts` (a dict) also fills in the quantize and decode shares:
    quant_bytes, quant_s, dec_bytes, dec_s."""
    import numpy as np
    import torch

    import oracle
    from paper_2609_35800_gb300 import workloads as wl

    mask = wl.protection_mask(w).numpy()
    B, H, T = w.batch, w.kv_heads, w.seq_len
    sigma = float(np.float32(1.0 / np.sqrt(128.0)))
    ns = oracle.salient_count(w.image, w.salient_permille) if w.salient_permille else 0

    def bits(t):
        return t.contiguous().view(torch.int16).numpy().view(np.uint16)

    secs = 0.0
    nbytes = 0
    outs = []
    q_secs = 0.0
    for l in range(n_layers):
        k, v = wl.layer_kv(w, l, "cpu")
        kb, vb = bits(k), bits(v)
        t0 = time.perf_counter()
        o = oracle.quantize_layer(kb, vb, w.img_start, w.image, w.base, w.bits, mask[l],
                                  int(w.keys_only), w.kivi_group_tokens, w.kivi_group_channels,
                                  w.kivi_residual, meta16=w.meta_bits == 32, n_salient=ns)
        secs += time.perf_counter() - t0
        q_secs += time.perf_counter() - t0
        nq = o["nq"] - ns  # coded tokens per quantized head
        code_tok = 128 * w.bits // 8
        n_prot = int(mask[l].sum())
        coded_heads_k = (H - n_prot)
        coded_heads_v = H if w.keys_only else (H - n_prot)
        shrink = 2 if w.meta_bits == 32 else 1  # binary16 pairs: half the fp32 pair bytes
        part = nq / max(o["nq"], 1)  # metadata of the coded tokens only
        meta_k = int(o["k_meta"][0, 0].nbytes * part) // shrink if coded_heads_k else 0
        meta_v = int(o["v_meta"][0, 0].nbytes * part) // shrink if coded_heads_v else 0
        written = B * (H * T * 512 - (coded_heads_k + coded_heads_v) * nq * 256
                       + coded_heads_k * (nq * code_tok + meta_k)
                       + coded_heads_v * (nq * code_tok + meta_v))
        nbytes += B * H * T * 512 + written
        outs.append(o)
    q_bytes = nbytes
    app_k = [[] for _ in range(n_layers)]
    app_v = [[] for _ in range(n_layers)]
    for s in range(n_steps):
        kn, vn = wl.step_new_kv(w, s, "cpu", n_layers)
        q = wl.step_query(w, s, "cpu", n_layers)
        knb, vnb, qb = bits(kn), bits(vn), bits(q)
        for l in range(n_layers):
            app_k[l].append((knb[l].astype(np.uint32) << 16).view(np.float32).astype(np.float64))
            app_v[l].append((vnb[l].astype(np.uint32) << 16).view(np.float32).astype(np.float64))
            K = np.concatenate([outs[l]["k_att"], np.stack(app_k[l], axis=2)], axis=2)
            V = np.concatenate([outs[l]["v_deq"].astype(np.float64), np.stack(app_v[l], axis=2)],
                               axis=2)
            t0 = time.perf_counter()
            oracle.attention_layer(qb[l], K, V, sigma)
            secs += time.perf_counter() - t0
            Tt = K.shape[2]
            # same per-token bytes as the packed cache the GPU reads
            nbytes += _decode_bytes_layer(w, mask[l], outs[l]["nq"], Tt - T, ns) + 2 * B * w.q_heads * 256
    threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    if parts is not None:
        parts.update(quant_bytes=q_bytes, quant_s=q_secs, dec_bytes=nbytes - q_bytes,
                     dec_s=secs - q_secs)
    return nbytes, secs, threads


def cpu_baseline_fields(w, n_layers, n_steps, parts):
    """The oracle's quantize GB/s and decode tokens/s from timed samples
    holding n_steps decode steps in all (decode tokens/s scaled to all layers
    when the sample holds fewer)."""
    dec_tok = w.batch * n_steps / parts["dec_s"] * (n_layers / w.layers) if parts["dec_s"] > 0 else None
    return {"quantize_GBps": round(parts["quant_bytes"] / parts["quant_s"] / 1e9, 4),
            "decode_GBps": round(parts["dec_bytes"] / parts["dec_s"] / 1e9, 4),
            "decode_tokens_per_s": round(dec_tok, 3) if dec_tok else None,
            "decode_tokens_per_s_basis": ("timed over all %d layers" % w.layers if n_layers == w.layers
                                          else "extrapolated from %d of %d layers" % (n_layers, w.layers)),
            "nproc": os.cpu_count(), "cpu_model": cpu_model()}


def _decode_bytes_layer(w, mask_row, nq, appended, ns=0):
    B, H, T = w.batch, w.kv_heads, w.seq_len
    code_tok = 128 * w.bits // 8
    pair = 4 if w.meta_bits == 32 else 8  # bytes of one {scale, zero}
    kmeta = (128 * pair // 32) if w.base == 1 else pair
    vmeta = 4 * pair if w.base == 1 else pair
    tot = 0
    for h in range(H):
        prot = bool(mask_row[h])
        if prot and not w.keys_only:
            tot += (T + appended) * 512
        elif prot:
            tot += (T - nq + ns + appended) * 512 + (nq - ns) * (256 + code_tok + vmeta)
        else:
            tot += (T - nq + ns + appended) * 512 + (nq - ns) * (2 * code_tok + kmeta + vmeta)
    return B * tot


def cpu_sample_plan(w):
    """One sample of the oracle: the whole workload step (every layer's
    quantization, then every decode step) on the small caches; the first layer
    and two decode steps on the large ones."""
    per_layer_tokens = w.batch * w.kv_heads * w.seq_len
    if per_layer_tokens <= 10000:
        return w.layers, w.decode_steps
    return 1, 2


def timed_oracle_samples(w, n_layers, n_steps, min_seconds=10.0, max_reps=50):
    """Repeat the oracle sample until at least min_seconds of timed oracle
    calls have accumulated (a bounded CPU baseline).  Returns (bytes, seconds,
    threads, repetitions, parts) summed over the repetitions."""
    tot_b, tot_s, reps, threads = 0, 0.0, 0, 1
    parts = {"quant_bytes": 0, "quant_s": 0.0, "dec_bytes": 0, "dec_s": 0.0}
    while reps < max_reps and (reps == 0 or tot_s < min_seconds):
        one = {}
        nb, secs, threads = oracle_sample(w, n_layers, n_steps, one)
        tot_b += nb
        tot_s += secs
        reps += 1
        for k in parts:
            parts[k] += one[k]
    return tot_b, tot_s, threads, reps, parts


def _workload(args):
    import dataclasses
    from paper_2609_35800_gb300 import workloads as wl
    w = wl.WORKLOADS[args.workload]
    if args.meta_bits != w.meta_bits:
        w = dataclasses.replace(w, meta_bits=args.meta_bits, name=w.name + "_meta%d" % args.meta_bits)
    if args.layers and args.layers != w.layers:
        w = dataclasses.replace(w, layers=args.layers, name=w.name + "_%dlayers" % args.layers)
    if args.bits and args.bits != w.bits:
        w = dataclasses.replace(w, bits=args.bits, name=w.name + "_%dbit" % args.bits)
    if args.salient_permille != w.salient_permille:
        w = dataclasses.replace(w, salient_permille=args.salient_permille,
                                name=w.name + "_salient%d" % args.salient_permille)
    return w


def workload_config(w):
    """The line's `config` (the same for both arms): the workload by name and shape."""
    from paper_2609_35800_gb300 import workloads as wl
    return {"workload": w.name, "layers": w.layers, "batch": w.batch,
            "q_heads": w.q_heads, "kv_heads": w.kv_heads,
            "tokens": "%d text + %d image + %d text" % (w.text_prefix, w.image, w.text_suffix),
            "base": ["minmax", "kivi", "akvq"][w.base], "bits": w.bits,
            "keys_only": w.keys_only, "protected_heads": int(wl.protection_mask(w).sum()),
            "decode_steps": w.decode_steps,
            "l2": "flushed (512 MiB write + read) before every timed launch group",
            "launch": "quantize: all layers per launch; each decode step: one launch appending the "
                      "new K/V and attending over all layers"}


def run_reference(args):
    from paper_2609_35800_gb300 import workloads as wl
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    w = _workload(args)
    n_layers, n_steps = cpu_sample_plan(w)
    vals = []
    tot_s = 0.0
    parts = {}
    for i in range(args.warmup + args.steps):
        nb, secs, threads = oracle_sample(w, n_layers, n_steps, parts)
        if i >= args.warmup:
            vals.append(nb / secs / 1e9)
            tot_s += secs
    value = statistics.median(vals)
    sample = ("%s: oracle quantize of %d layer(s) then %d decode step(s) of fp64 attention over "
              "them; timed oracle calls only" % (w.name, n_layers, n_steps))
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "GB/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(1000 * tot_s / max(1, args.steps), 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "fp32/fp64", "data": "synthetic",
        "config": workload_config(w),
        "cpu_baseline": dict({"value": round(value, 4), "unit": "GB/s", "cores": threads,
                              "kind": "oracle", "sample": sample},
                             **cpu_baseline_fields(w, n_layers, n_steps, parts)),
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

def run_gpu(args):
    import torch

    import paper_2609_35800_gb300 as hg
    from paper_2609_35800_gb300 import build, workloads as wl
    from paper_2609_35800_gb300.runner import CacheRunner

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    if rank == 0:
        build.build()
    if dist is not None:
        dist.barrier()
    hg.library()

    w = _workload(args)
    dev = "cuda:%d" % local
    stream = torch.cuda.current_stream()
    runner = CacheRunner(w, device=dev)
    L, S = w.layers, w.decode_steps
    # resident inputs of one step
    prefill = [wl.layer_kv(w, l, dev) for l in range(L)]
    ks = [k for k, _ in prefill]
    vs = [v for _, v in prefill]
    qs = [wl.step_query(w, s, dev) for s in range(S)]
    news = [wl.step_new_kv(w, s, dev) for s in range(S)]
    out = torch.empty_like(qs[0])
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    sigma = 0.0
    quant_b, dec_b, app_b = geometry_bytes(runner)
    step_bytes = quant_b + sum(dec_b) + S * app_b
    # quantize: per 64 layers one launch (two for the AKVQ- and KIVI-style bases:
    # keys, values), preceded by the salient-token selection when on
    q_launches = (L + 63) // 64 * ((2 if w.base in (wl.BASE_AKVQ, wl.BASE_KIVI) else 1)
                                   + (1 if (w.salient_permille > 0 and w.image > 0) else 0))
    launches_per_step = q_launches + S * ((L + 63) // 64)

    def cushion():
        flush.zero_()            # evict L2 (write a buffer larger than L2) ...
        flush.sum()              # ... and read it back so the evicted lines are clean
        torch.cuda._sleep(200000)  # keep the stream busy while the host enqueues the group

    def one_step(record):
        ev = []
        cushion()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for l0 in range(0, L, 64):
            n = min(64, L - l0)
            hg.hg_quantize_kv(runner.cache, l0, ks[l0:l0 + n], vs[l0:l0 + n], stream)
        e1.record(stream)
        ev.append(("quant", e0, e1))
        hg.hg_cache_reset_appended(runner.cache)
        for s in range(S):
            cushion()
            a0, a1 = (torch.cuda.Event(enable_timing=True) for _ in range(2))
            a0.record(stream)
            hg.hg_decode_step(runner.cache, 0, L, qs[s], news[s][0], news[s][1], out, sigma,
                              runner.ws, runner.ws_bytes, stream)
            a1.record(stream)
            ev.append(("decode", a0, a1))
        if record is not None:
            record.append(ev)

    for _ in range(args.warmup):
        one_step(None)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    records = []
    with ClockSampler(local) as clk:
        t_wall = time.perf_counter()
        for _ in range(args.steps):
            one_step(records)
        torch.cuda.synchronize()
        t_wall = time.perf_counter() - t_wall
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()

    per = {"quant": [], "decode": []}
    step_ms = []
    for ev in records:
        tot = 0.0
        for kind, a, b in ev:
            ms = a.elapsed_time(b)
            per[kind].append(ms)
            tot += ms
        step_ms.append(tot)
    ms_step = max_over_ranks(sum(step_ms) / len(step_ms), dist, dev)
    value = whole_job_gbs(world, step_bytes, ms_step)

    quant_ms = statistics.mean(per["quant"])
    dec_ms = statistics.mean(per["decode"])
    dec_bytes_mean = (sum(dec_b) + S * app_b) / S
    tok_s = world * w.batch * S / (sum(per["decode"]) / args.steps * 1e-3)

    peaks, peak_src = measured_peaks()
    peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    achieved = dec_bytes_mean / (dec_ms * 1e-3) / 1e9
    traffic = profiled_traffic(w.name)

    extra = None
    if not args.no_variants:
        extra = decode_variants(args, runner, w, qs, news, dec_b, app_b, cushion, stream)

    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, runner, w, prefill, qs, news, step_bytes, dev, stream)

    try:
        deq = time_dequantize(runner, w, dec_b, dev, cushion, stream)
    except Exception as exc:  # a side measurement never costs the line
        deq = {"error": "%s: %s" % (type(exc).__name__, exc)}
    try:
        floors = measure_floors(int(dec_bytes_mean), cushion, stream, dev)
    except Exception as exc:
        floors = {"error": "%s: %s" % (type(exc).__name__, exc)}

    line = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16/fp16 MMA operands, fp32 accumulate; fp32 quantizer", "data": "synthetic",
        "config": workload_config(w),
        "pct_of_8TBps": round(100 * value / NOMINAL_HBM_GBS, 2),
        "pct_of_measured_hbm": round(100 * value / peak, 2),
        "decode_tokens_per_s": round(tok_s, 1),
        "kernels": {
            "quantize": {"ms": round(quant_ms, 4), "GBps": round(quant_b / quant_ms / 1e6, 1)},
            "decode_step (append + attention, one launch)": {"ms": round(dec_ms, 4),
                                                               "GBps": round(achieved, 1)},
            "dequantize (all layers, not part of the step)": deq,
        },
        "step_bytes": step_bytes,
        "wall_s_timed_region": round(t_wall, 4),
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": traffic,
                     "kernel": "decode_kernel (hg_decode_step)",
                     "peak_source": peak_src + " hbm_gbs (burst copy)"},
        "floors": floors,
        "clocks": clk.summary(),
        "gpu_launches": launches_per_step * args.steps,
    }
    if extra is not None:
        line["decode_variants"] = extra
    if e2e is not None:
        line["e2e"] = e2e
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n_layers, n_steps = cpu_sample_plan(w)
        nb, secs, threads, reps, parts = timed_oracle_samples(w, n_layers, n_steps)
        line["cpu_baseline"] = dict({
            "value": round(nb / secs / 1e9, 4), "unit": "GB/s", "cores": threads, "kind": "oracle",
            "sample": "%s: %d repetition(s) of oracle quantize of %d layer(s) then %d decode step(s) of "
                      "fp64 attention over them, %.1f s of timed oracle calls" % (w.name, reps, n_layers,
                                                                                   n_steps, secs)},
            **cpu_baseline_fields(w, n_layers, n_steps * reps, parts))
    if rank == 0:
        print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()
    return 0


def decode_variants(args, runner, w, qs, news, dec_b, app_b, cushion, stream):
    """Two other ways to launch the same decode steps, reported beside the
    headline (which they do not change): one launch per layer (append and
    attention of a single layer each), L2 flushed before every step; and the
    whole decode loop captured in one CUDA graph and replayed (launch costs
    gone; the cache stays in L2 between steps, as it would when nothing else
    runs between decode steps)."""
    import torch

    import paper_2609_35800_gb300 as hg
    L, S = w.layers, w.decode_steps
    out = torch.empty_like(qs[0])
    dec_bytes_mean = (sum(dec_b) + S * app_b) / S
    res = {}
    # one launch per layer
    hg.hg_cache_reset_appended(runner.cache)
    n_steps = min(S, 8)
    times = []
    for st in range(n_steps):
        cushion()
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for l in range(L):
            hg.hg_decode_step(runner.cache, l, 1, qs[st][l], news[st][0][l], news[st][1][l], out[l],
                              0.0, runner.ws, runner.ws_bytes, stream)
        a1.record(stream)
        times.append((a0, a1))
    torch.cuda.synchronize()
    ms = statistics.mean(a.elapsed_time(b) for a, b in times)
    res["per_layer_launches"] = {"ms_per_decode_step": round(ms, 4), "launches_per_step": L,
                                 "GBps": round(dec_bytes_mean / (ms * 1e-3) / 1e9, 1),
                                 "steps_timed": n_steps, "l2": "flushed before every step"}
    # append and attention as two launches per step (hg_append_kv, then
    # hg_decode_attention), both over all layers
    hg.hg_cache_reset_appended(runner.cache)
    times = []
    for st in range(n_steps):
        cushion()
        a0, a1, a2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
        a0.record(stream)
        hg.hg_append_kv(runner.cache, 0, L, news[st][0], news[st][1], stream)
        a1.record(stream)
        hg.hg_decode_attention(runner.cache, 0, L, qs[st], out, 0.0, runner.ws, runner.ws_bytes, stream)
        a2.record(stream)
        times.append((a0, a1, a2))
    torch.cuda.synchronize()
    app_ms = statistics.mean(a.elapsed_time(b) for a, b, _ in times)
    att_ms = statistics.mean(b.elapsed_time(c) for _, b, c in times)
    res["append_then_attention"] = {
        "append_ms": round(app_ms, 4), "append_GBps": round(app_b / (app_ms * 1e-3) / 1e9, 1),
        "attention_ms": round(att_ms, 4),
        "attention_GBps": round((dec_bytes_mean - app_b) / (att_ms * 1e-3) / 1e9, 1),
        "steps_timed": n_steps, "l2": "flushed before every step"}
    # the decode loop as one CUDA graph (layer-batched launches)
    hg.hg_cache_reset_appended(runner.cache)
    graph = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        with torch.cuda.graph(graph, stream=side):
            cap = torch.cuda.current_stream()
            for st in range(S):
                hg.hg_decode_step(runner.cache, 0, L, qs[st], news[st][0], news[st][1], out, 0.0,
                                  runner.ws, runner.ws_bytes, cap)
    torch.cuda.current_stream().wait_stream(side)
    graph.replay()
    torch.cuda.synchronize()
    reps = []
    for _ in range(5):
        cushion()
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        graph.replay()
        a1.record(stream)
        torch.cuda.synchronize()
        reps.append(a0.elapsed_time(a1) / S)
    best, med = min(reps), statistics.median(reps)
    res["graph_replay"] = {"ms_per_decode_step_best": round(best, 4),
                           "ms_per_decode_step_median": round(med, 4),
                           "GBps_best": round(dec_bytes_mean / (best * 1e-3) / 1e9, 1),
                           "decode_tokens_per_s_best": round(w.batch / (best * 1e-3), 1),
                           "l2": "flushed before each replay of the %d-step loop only" % S}
    hg.hg_cache_reset_appended(runner.cache)
    return res


def measure_floors(nbytes, cushion, stream, dev, reps=10):
    """Fixed costs of an event-timed launch on this device, for reading the
    decode fraction: two events with nothing between them, one near-empty
    kernel, and a plain read of the decode step's byte count by torch's own
    reduction (the same L2 flush before each).  Medians in microseconds."""
    import torch
    buf = torch.ones(max(1, nbytes // 4), dtype=torch.int32, device=dev)

    def timed(fn):
        ts = []
        for _ in range(reps):
            cushion()
            a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a0.record(stream)
            fn()
            a1.record(stream)
            ts.append((a0, a1))
        torch.cuda.synchronize()
        return statistics.median(a.elapsed_time(b) * 1000.0 for a, b in ts)

    events = timed(lambda: None)
    empty = timed(lambda: torch.cuda._sleep(0))
    read = timed(lambda: buf.max())
    return {"events_only_us": round(events, 2), "empty_kernel_us": round(empty, 2),
            "read_same_bytes_us": round(read, 2), "read_bytes": buf.numel() * 4,
            "read_GBps": round(buf.numel() * 4 / (read * 1e-6) / 1e9, 1),
            "how": "CUDA events on the launching stream after the same L2 flush; the read is "
                   "torch.max over an int32 buffer of the decode step's byte count"}


def time_dequantize(runner, w, dec_b, dev, cushion, stream, reps=3, budget_bytes=4 << 30):
    """Reconstruction of every layer as BF16 (Sec. 4: code * scale + zero, the
    AKVQ-style keys rotated back; text, protected and appended entries copied):
    one launch over as many layers as fit `budget_bytes` of output per tensor
    (all of them on the smaller caches), L2 flushed before each group of
    launches.  Bytes: the cache entries a decode step reads (codes, metadata,
    BF16 rows) plus the two BF16 outputs [layers][B][H_kv][T + appended][128]."""
    import torch

    import paper_2609_35800_gb300 as hg
    L, B, H, Hq = w.layers, w.batch, w.kv_heads, w.q_heads
    app = hg.hg_cache_appended(runner.cache, 0)
    q_rows = L * B * Hq * 256
    dec_static = dec_b[0] - L * H * B * 512 - 2 * q_rows  # cache bytes without appended rows
    tt = w.seq_len + app
    nbytes = dec_static + L * H * B * app * 512 + L * 2 * B * H * tt * 256
    per_layer = B * H * tt * 256
    chunk = max(1, min(L, budget_bytes // per_layer))
    k16 = torch.empty((chunk, B, H, tt, 128), dtype=torch.bfloat16, device=dev)
    v16 = torch.empty_like(k16)
    times = []
    for _ in range(reps):
        cushion()
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for l0 in range(0, L, chunk):
            n = min(chunk, L - l0)
            hg.hg_dequantize_kv(runner.cache, l0, n, k16, v16, False, stream)
        a1.record(stream)
        times.append((a0, a1))
    torch.cuda.synchronize()
    ms = statistics.mean(a.elapsed_time(b) for a, b in times)
    return {"ms": round(ms, 4), "GBps": round(nbytes / (ms * 1e-3) / 1e9, 1),
            "launches": (L + chunk - 1) // chunk, "layers_per_launch": chunk,
            "appended": app, "bytes": nbytes, "l2": "flushed before each group of launches"}


def run_e2e(args, runner, w, prefill, qs, news, step_bytes, dev, stream, n_chunks=4):
    """Same step driven from pinned HOST buffers through the C ABI.

    The prefill K and V of all layers sit in one pinned buffer each; they are
    copied to the device in `n_chunks` layer groups on a copy stream, and each
    group is quantized as soon as its copy has landed (the copy engine moves
    the whole prefill while the quantizer works on the groups already there).
    Each decode step's query, new keys and new values sit in one pinned buffer
    and its attention output goes to another: the decode kernel reads the
    inputs from, and writes the output to, host memory directly (pinned host
    memory is addressable from the device), so a step costs no copy-engine
    round trip.  h2d / d2h bytes count everything that crosses the link."""
    import torch

    import paper_2609_35800_gb300 as hg
    L, S = w.layers, w.decode_steps
    hk = torch.stack([k for k, _ in prefill]).cpu().pin_memory()
    hv = torch.stack([v for _, v in prefill]).cpu().pin_memory()
    nq, nk = qs[0].numel(), news[0][0].numel()
    hin = torch.empty((S, nq + 2 * nk), dtype=qs[0].dtype).pin_memory()
    for st in range(S):
        hin[st, :nq].copy_(qs[st].reshape(-1).cpu())
        hin[st, nq:nq + nk].copy_(news[st][0].reshape(-1).cpu())
        hin[st, nq + nk:].copy_(news[st][1].reshape(-1).cpu())
    hout = torch.empty((S,) + tuple(qs[0].shape), dtype=qs[0].dtype).pin_memory()
    dk = torch.empty_like(hk, device=dev)
    dv = torch.empty_like(hv, device=dev)
    dks = [dk[l] for l in range(L)]
    dvs = [dv[l] for l in range(L)]
    h2d = (hk.numel() + hv.numel() + hin.numel()) * 2
    d2h = hout.numel() * 2
    per = (L + n_chunks - 1) // n_chunks
    groups = [(l0, min(L, l0 + per)) for l0 in range(0, L, per)]
    copy_stream = torch.cuda.Stream(device=dev)
    esz = qs[0].element_size()

    def step():
        copy_stream.wait_stream(torch.cuda.current_stream())
        landed = []
        with torch.cuda.stream(copy_stream):
            for l0, l1 in groups:
                dk[l0:l1].copy_(hk[l0:l1], non_blocking=True)
                dv[l0:l1].copy_(hv[l0:l1], non_blocking=True)
                ev = torch.cuda.Event()
                ev.record(copy_stream)
                landed.append(ev)
        for (l0, l1), ev in zip(groups, landed):
            stream.wait_event(ev)
            for g0 in range(l0, l1, 64):
                n = min(64, l1 - g0)
                hg.hg_quantize_kv(runner.cache, g0, dks[g0:g0 + n], dvs[g0:g0 + n], stream)
        for st in range(S):
            base = hin[st].data_ptr()
            hg.hg_decode_step(runner.cache, 0, L, base, base + nq * esz, base + (nq + nk) * esz,
                              hout[st].data_ptr(), 0.0, runner.ws, runner.ws_bytes, stream)

    for _ in range(max(1, args.warmup)):
        step()
    torch.cuda.synchronize()
    times = []
    for _ in range(args.steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step()
        e1.record(stream)
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    hg.hg_cache_reset_appended(runner.cache)
    ms = statistics.mean(times)
    return {"value": round(step_bytes / (ms * 1e-3) / 1e9, 2), "unit": "GB/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": round(ms, 4),
            "prefill": "%d layer groups copied on a copy stream, each quantized as it lands" % len(groups),
            "decode_inputs_outputs": "read and written by the decode kernel in pinned host memory"}


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())

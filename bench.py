"""Throughput of the LM-GC encode path on GB300 (one JSON line on rank 0).

Workload (default, the largest single-GPU configuration): gradients of a seeded random-init
4-layer ConvNet (298,954 values, 3x32x32 Gaussian inputs, batch 64), serialised as 8 hex digits +
a space per value, coded with a Llama-2-7B-shaped model (32 layers, d 4096, 32 heads MHA, FFN
11008, vocab 32000, random-init bf16 weights) over 4096-token windows, 32 windows per model
batch, 24-bit integer CDFs. One step = lmgc_encode of one batch: 14,563 values (131,067 tokens,
32 windows) through serialise -> model -> CDF pairs -> range coder -> container. Step k encodes
slice k mod 20 of the gradient; all slices are resident in HBM before timing. The line also
carries the TinyLlama-shaped step (22 layers, d 2048, 32/4 heads, FFN 5632, 2048-token windows,
64 per batch) under "tinyllama_step".

value     raw-gradient MB/s (4 bytes per value) over all ranks, device buffers, CUDA events
e2e       the same through lmgc_encode_host (pinned host buffers; H2D + D2H inside the region)
roofline  the GEMM class (the dominant kernel): algorithmic flops / summed CUDA-event time of its
          launches in the timed region, against the measured sustained bf16 peak
stages    the same per kernel class (HBM-bound classes against the measured HBM copy bandwidth)
cpu_baseline / --impl reference: the CPU oracle (test infrastructure) on a bounded sample.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "raw gradient MB/s encoded (1 GB300); LM tensor-pipe % of bf16 peak; coder HBM GB/s"
DEFAULT_WORKLOAD = "convnet-llama2-7b"
WORKLOADS = ("convnet-tinyllama", "tiny", "convnet-llama2-7b", "lossy-tinyllama", "laplace-tinyllama",
             "quant16-tinyllama", "quant1-tinyllama", "sparse50-tinyllama", "sparse25-tinyllama",
             "alpha-tinyllama")


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(p))
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sus=d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                    src="measured")
    except Exception:
        return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")


class Clocks:
    """nvidia-smi samples every 200 ms during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"], stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def workload(name: str):
    from paper_2409_17836_gb300 import configs, inputs

    if name == "convnet-tinyllama":
        return configs.TINYLLAMA, inputs.convnet_gradient(0)
    if name == "convnet-llama2-7b":
        return configs.LLAMA2_7B, inputs.convnet_gradient(0)
    if name == "lossy-tinyllama":
        return configs.TINYLLAMA_LOSSY, inputs.lossy_codes(inputs.convnet_gradient(0))
    if name == "tiny":
        return configs.TINY, inputs.tiny_gradient(0)
    if name == "laplace-tinyllama":  # 64M-value Laplace mixture; window batch set by --batch-windows
        return configs.TINYLLAMA, inputs.laplace_gradient()
    # Sec. 5.4 compatibility settings one at a time: Eq. 4 indices of every value (16 bits as
    # big-endian byte pairs, one separator per index; 1 bit as one byte each), or the top 50% / 25%
    # of |v| still as fp32
    if name in ("quant16-tinyllama", "quant1-tinyllama"):
        b, group = inputs.code_bytes(inputs.quantized_codes(inputs.convnet_gradient(0), 16 if "16" in name else 1))
        return configs.with_(configs.TINYLLAMA, input_kind=1, byte_group=group), b
    if name in ("sparse50-tinyllama", "sparse25-tinyllama"):
        return configs.TINYLLAMA, inputs.sparsified(inputs.convnet_gradient(0), 0.5 if "50" in name else 0.25)
    if name == "alpha-tinyllama":  # integer CDFs over the 17 ids the space-separated stream can emit
        return configs.with_(configs.TINYLLAMA, alphabet=1), inputs.convnet_gradient(0)
    raise ValueError(name)


def values_for_tokens(count, n_max: int, budget: int) -> int:
    """The most values (<= n_max) whose serialisation fits in `budget` tokens; count(n) = tokens."""
    lo, hi = 0, n_max
    while lo < hi:
        mid = (lo + hi + 1) // 2
        if count(mid) <= budget:
            lo = mid
        else:
            hi = mid - 1
    return lo


def run_full(args, cfg, ctx, vals):
    """One lmgc_encode of the whole workload (inputs resident on the device), timed with CUDA
    events; then the first, middle and last windows are decoded (KV-cached) and compared with the
    serialised input tokens."""
    import numpy as np
    import torch

    import oracle as O
    from paper_2409_17836_gb300 import lmgc as L

    d = torch.from_numpy(vals.view(np.int32) if vals.dtype == np.float32 else vals).cuda()
    out = torch.empty(L.lmgc_encode_bound(ctx, vals.size), dtype=torch.uint8, device="cuda")
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    with Clocks(torch.cuda.current_device()) as clk:
        e0.record()
        buf = L.lmgc_encode(ctx, d, out)
        e1.record()
        torch.cuda.synchronize()
    sec = e0.elapsed_time(e1) / 1e3
    W = cfg.window
    n_tok = L.lmgc_serial_tokens(ctx, vals.size)
    n_win = -(-n_tok // W)
    ids = [0, n_win // 2, n_win - 1]
    toks = L.lmgc_decode(ctx, buf, ids).cpu().numpy().view(np.uint16)
    ok = True
    tpv = ctx.tpv
    whole = None if tpv else O.serialize(vals, cfg.sep_mode, cfg.byte_group, cfg.byte_order)
    for i, w in enumerate(ids):
        n = min(W, n_tok - w * W)
        if tpv:
            v0, v1 = (w * W) // tpv, -(-min(n_tok, (w + 1) * W) // tpv)
            ref = O.serialize(vals[v0:v1], cfg.sep_mode, cfg.byte_group, cfg.byte_order)[w * W - v0 * tpv:][:n]
        else:
            ref = whole[w * W: w * W + n]
        ok = ok and bool(np.array_equal(toks[i, :n], ref))
    bpv = 4 if vals.dtype == np.float32 else 1
    print(json.dumps({"mode": "full", "workload": args.workload, "values": int(vals.size), "windows": int(n_win),
                      "batch_windows": cfg.batch_windows, "seconds": sec,
                      "value": vals.size * bpv / sec / 1e6, "unit": "MB/s",
                      "container_bytes": int(buf.numel()),
                      "compression_rate_pct": 100.0 * buf.numel() / (vals.size * bpv),
                      "decoded_windows": ids, "decoded_match": ok, "clocks": clk.summary()}), flush=True)
    ctx.close()
    return 0 if ok else 1


def run_decode(args, cfg, ctx, vals):
    """lmgc_decode of every window of an encoded stream (--decode-windows full windows; default as
    many as one decode batch takes, that is as many as the library's KV cache budget holds, at
    most the whole stream), timed with CUDA events around the call; the restored tokens are
    compared with the serialised input."""
    import numpy as np
    import torch

    import oracle as O
    from paper_2409_17836_gb300 import lmgc as L

    W = cfg.window
    n_all = -(-L.lmgc_serial_tokens(ctx, vals.size) // W)
    # (the encode below takes a little device memory of its own: keep 5% of the batch as slack so
    # that the decode still runs as one batch)
    n_dec = args.decode_windows or max(1, min(n_all, (L.lmgc_decode_batch_windows(ctx) * 19) // 20))
    n = values_for_tokens(lambda m: L.lmgc_serial_tokens(ctx, m), vals.size, n_dec * W)
    v = vals[:n]
    d = torch.from_numpy(v.view(np.int32) if v.dtype == np.float32 else v).cuda()
    buf = L.lmgc_encode(ctx, d)
    n_tok = L.lmgc_serial_tokens(ctx, n)
    n_win = -(-n_tok // W)
    ids = list(range(n_win))
    L.lmgc_decode(ctx, buf, ids[:1])  # warm-up
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    with Clocks(torch.cuda.current_device()) as clk:
        e0.record()
        toks = L.lmgc_decode(ctx, buf, ids)
        e1.record()
        torch.cuda.synchronize()
    sec = e0.elapsed_time(e1) / 1e3
    # the same decode again with per-class kernel timing (CUDA events around each launch)
    L.lmgc_profile(ctx, True)
    L.lmgc_decode(ctx, buf, ids)
    torch.cuda.synchronize()
    st = L.lmgc_kernel_stats(ctx)
    L.lmgc_profile(ctx, False)
    classes = {k: {"launches": x["launches"], "ms": round(x["ms"], 1)} for k, x in st.items() if x["launches"]}
    ref = O.serialize(v, cfg.sep_mode, cfg.byte_group, cfg.byte_order)
    got = toks.cpu().numpy().view(np.uint16).reshape(-1)[:n_tok]
    print(json.dumps({"mode": "decode", "workload": args.workload, "windows": n_win, "tokens": n_tok,
                      "seconds": sec, "tokens_per_s": n_tok / sec, "ms_per_position": 1e3 * sec / W,
                      "match": bool(np.array_equal(got, ref)), "clocks": clk.summary(),
                      "classes_profiled_run": classes}), flush=True)
    ctx.close()
    return 0


def oracle_sample(cfg, vals, positions: int, win: int, threads: int):
    """Oracle encode of the first `positions` tokens of window `win` (model + CDF + coder)."""
    import numpy as np

    import oracle as O

    oc = O.OracleConfig(n_layers=cfg.n_layers, d_model=cfg.d_model, n_heads=cfg.n_heads, n_kv_heads=cfg.n_kv_heads,
                        d_ffn=cfg.d_ffn, vocab=cfg.vocab, bf16=cfg.dtype == 1, window=cfg.window,
                        cdf_bits=cfg.cdf_bits, weight_seed=cfg.weight_seed, init_std=cfg.init_std,
                        sep_mode=cfg.sep_mode, input_kind=cfg.input_kind, n_threads=threads,
                        byte_group=cfg.byte_group, byte_order=cfg.byte_order, alphabet=cfg.alphabet)
    tok = O.serialize(vals, cfg.sep_mode, cfg.byte_group, cfg.byte_order)
    W = cfg.window
    seg = tok[win * W: win * W + W]
    t0 = time.perf_counter()
    st, fr, _ = O.window_pairs(oc, seg, min(positions, seg.size))
    O.range_encode(st, fr, cfg.cdf_bits)
    dt = time.perf_counter() - t0
    return dt, min(positions, seg.size)


def cpu_baseline(cfg, vals, tpv: float, bpv: int, target_s: float) -> dict:
    """The oracle as it stands on the host's cores: a prefix of window 0 sized for about target_s
    seconds with every core, then a prefix sized for about target_s / 4 on one thread. The
    one-thread figure is left out when even its 4-position calibration would take longer than
    target_s (estimated as the all-core calibration times the core count: the Llama-2-7B shape)."""
    threads = max(1, len(os.sched_getaffinity(0)))
    what = "oracle encode (fp64 model forward, integer CDF, range coder) of the first {} tokens of window 0, {:.1f} s"
    dt4, n4 = oracle_sample(cfg, vals, 4, 0, threads)
    positions = int(max(4, min(cfg.window, target_s / max(dt4 / n4, 1e-6))))
    dt, n = oracle_sample(cfg, vals, positions, 0, threads)
    res = {"value": n / tpv * bpv / dt / 1e6, "unit": "MB/s", "cores": threads, "kind": "oracle",
           "sample": what.format(n, dt)}
    est1 = dt4 * threads
    if est1 > target_s:
        res["single_thread"] = {"skipped": f"a 4-position calibration on one thread would take about {est1:.0f} s"}
        return res
    dt1, n1 = oracle_sample(cfg, vals, 4, 0, 1)
    positions = int(max(4, min(cfg.window, target_s / 4 / max(dt1 / n1, 1e-6))))
    dt1, n1 = oracle_sample(cfg, vals, positions, 0, 1)
    res["single_thread"] = {"value": n1 / tpv * bpv / dt1 / 1e6, "unit": "MB/s", "cores": 1,
                            "sample": what.format(n1, dt1)}
    return res


def microbenchmarks(L, ctx, pk, reps: int = 3, coder_windows: int = 1 << 20) -> dict:
    """HBM-bound stages at sizes where bandwidth, not launch latency, decides: the serialiser on
    the 64M-value Laplace mixture (default layout, and byte groups of 3 that cross values), and
    the coder alone (lmgc_range_encode_tiled, pairs in the window tiles the encode path uses) on
    2^20 windows x 2048 tokens (the 64M-value sweep's coder microbenchmark) of seeded random
    integer CDFs over vocab 32000 at P = 24 (half the symbols the row's most likely); ctx supplies
    the integer CDFs (any context with vocab 32000 and P = 24)."""
    import numpy as np
    import torch

    from paper_2409_17836_gb300 import configs, inputs

    out = {}
    vals = inputs.laplace_gradient()
    d = torch.from_numpy(vals.view(np.int32)).cuda()
    sctx = L.Context(configs.TINY)  # fp32 values, one group per value, H_s
    tok = torch.empty(L.lmgc_serial_tokens(sctx, d.numel()), dtype=torch.int16, device="cuda")
    L.lmgc_serialize(sctx, d, tok)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        L.lmgc_serialize(sctx, d, tok)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    nbytes = d.numel() * 4 + tok.numel() * 2
    out["serialize"] = {"values": d.numel(), "ms": ms, "bytes": nbytes, "achieved": nbytes / ms / 1e6,
                        "unit": "GB/s", "frac": nbytes / ms / 1e6 / pk["hbm"]}
    sctx.close()
    del tok
    # the byte-grouped layout (Sec. 5.3): 3 bytes per group, fp32 bytes least significant first
    gctx = L.Context(configs.with_(configs.TINY, byte_group=3, byte_order=1))
    tok = torch.empty(L.lmgc_serial_tokens(gctx, d.numel()), dtype=torch.int16, device="cuda")
    L.lmgc_serialize(gctx, d, tok)
    torch.cuda.synchronize()
    e0.record()
    for _ in range(reps):
        L.lmgc_serialize(gctx, d, tok)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    nbytes = d.numel() * 4 + tok.numel() * 2
    out["serialize_grouped"] = {"values": d.numel(), "byte_group": 3, "byte_order": 1, "ms": ms, "bytes": nbytes,
                                "achieved": nbytes / ms / 1e6, "unit": "GB/s", "frac": nbytes / ms / 1e6 / pk["hbm"]}
    gctx.close()
    del d, tok
    V, P, W, n_win = 32000, 24, 2048, coder_windows
    g = torch.Generator(device="cuda").manual_seed(5)
    z = torch.randn(256, V, generator=g, device="cuda") * torch.linspace(0.3, 6.0, 256, device="cuda")[:, None]
    cdf = L.lmgc_quantize_cdf(ctx, z).long()
    likely = torch.argmax(cdf[:, 1:] - cdf[:, :-1], dim=1)
    # window tiles, the encode path's layout: [window block][position group][window][position]
    assert n_win % 32 == 0 and W % 8 == 0
    NB, G = n_win // 32, W // 8
    start = torch.empty((NB, G, 32, 8), dtype=torch.int32, device="cuda")
    freq = torch.empty_like(start)
    step = min(NB, 1 << 10)  # 32,768 windows at a time
    for b0 in range(0, NB, step):
        nb = min(step, NB - b0)
        row = torch.randint(0, 256, (W, nb * 32), generator=g, device="cuda")
        sym = torch.randint(0, V, (W, nb * 32), generator=g, device="cuda")
        sym = torch.where(torch.rand((W, nb * 32), generator=g, device="cuda") < 0.5, likely[row], sym)
        st = cdf[row, sym]
        fr = cdf[row, sym + 1] - st
        # [position][window] -> [block][group][window in block][position in group]
        start[b0:b0 + nb] = st.int().view(G, 8, nb, 32).permute(2, 0, 3, 1)
        freq[b0:b0 + nb] = fr.int().view(G, 8, nb, 32).permute(2, 0, 3, 1)
        del row, sym, st, fr
    # "range_encode": the coder as the encode path runs it (its pairs, valid by construction, are
    # not checked again); "range_encode_validated": the same with every pair checked, as for a
    # caller's pairs. The codes must be identical.
    for key, validate in (("range_encode", False), ("range_encode_validated", True)):
        payload, _ = L.lmgc_range_encode_tiled(start, freq, P, n_win, W, None, validate=validate)
        torch.cuda.synchronize()
        L.lmgc_profile(None, True)
        for _ in range(reps):
            payload, _ = L.lmgc_range_encode_tiled(start, freq, P, n_win, W, None, out=payload, validate=validate)
        st = L.lmgc_kernel_stats(None)["range_encode"]
        L.lmgc_profile(None, False)
        kms = st["ms"] / max(1, st["launches"])
        rd = 8.0 * W * n_win
        wr = float(payload.numel())
        out[key] = {"windows": n_win, "tokens": W * n_win, "ms": kms, "read_bytes": rd, "write_bytes": wr,
                    "bits_per_token": 8.0 * wr / (W * n_win), "achieved": (rd + wr) / kms / 1e6,
                    "unit": "GB/s", "frac": (rd + wr) / kms / 1e6 / pk["hbm"],
                    "tokens_per_s": W * n_win / (kms / 1e3)}
        if validate:
            same = torch.equal(payload, ref_payload)
            out[key]["codes_equal_unchecked"] = bool(same)
            if not same:
                raise RuntimeError("coder microbenchmark: checked and unchecked codes differ")
        else:
            ref_payload = payload.clone()
    del start, freq, payload, ref_payload
    torch.cuda.empty_cache()
    return out


def micro_run(L, configs, pk, coder_windows: int) -> dict:
    """The microbenchmarks with a small vocab-32000, P = 24 context (one layer, one window per
    batch) that only supplies the coder's integer CDFs."""
    ctx = L.Context(configs.with_(configs.TINYLLAMA, n_layers=1, batch_windows=1))
    try:
        return microbenchmarks(L, ctx, pk, coder_windows=coder_windows)
    finally:
        ctx.close()


def profiled_traffic(workload: str, kernel: str, work_per_launch: float):
    """DRAM bytes per launch of a kernel class, scaled from a small-case ncu capture of the same
    kernels (profiles/traffic_<workload>-small.md: DRAM read + write bytes and algorithmic work
    summed over the captured launches) by the algorithmic work of one launch here; None when there
    is no capture. The scaling holds for the GEMMs, whose operand and output bytes grow with the
    rows processed (the weight is read once per group of row tiles in both cases)."""
    path = os.path.join(ROOT, "profiles", f"traffic_{workload}-small.md")
    try:
        text = open(path).read()
        block = json.loads(text.split("```json", 1)[1].split("```", 1)[0])[kernel]
        per_work = block["dram_bytes"] / block["work"]
        return per_work * work_per_launch, os.path.relpath(path, ROOT)
    except Exception:
        return None, None


def bytes_per_value(cfg) -> int:
    return 4 if cfg.input_kind == 0 else 1


def run_reference(args):
    """The CPU oracle as the reference arm: each step encodes a bounded prefix of one window."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle as O

    O.lib()
    cfg, vals = workload(args.workload)
    threads = max(1, len(os.sched_getaffinity(0)))
    n_tok = O.serial_tokens(cfg.input_kind, cfg.sep_mode, vals.size, cfg.byte_group, cfg.byte_order)
    tpv = n_tok / vals.size  # tokens per value over the workload
    positions = args.ref_positions
    n_win = -(-n_tok // cfg.window)
    for i in range(args.warmup):
        oracle_sample(cfg, vals, 2, i % n_win, threads)
    total_t, total_tok = 0.0, 0
    for k in range(args.steps):
        dt, n = oracle_sample(cfg, vals, positions, k % n_win, threads)
        total_t += dt
        total_tok += n
    mbs = total_tok / tpv * bytes_per_value(cfg) / total_t / 1e6
    sample = (f"oracle encode of the first {positions} tokens of one window per step (model forward over those "
              f"positions in fp64, integer CDF, range coder), {args.steps} steps")
    out = {"impl": "reference", "metric": METRIC, "value": mbs, "unit": "MB/s", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total_t / args.steps,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": args.workload, "window": cfg.window, "batch_windows": cfg.batch_windows},
           "cpu_baseline": {"value": mbs, "unit": "MB/s", "cores": threads, "kind": "oracle", "sample": sample},
           "e2e": {"value": mbs, "unit": "MB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def model_name(cfg) -> str:
    return f"{cfg.n_layers}L d{cfg.d_model} {cfg.n_heads}/{cfg.n_kv_heads}h ffn{cfg.d_ffn} V{cfg.vocab}"


def measure_steps(L, ctx, cfg, vals, args, world, rank, local, pk, name, e2e=True) -> dict:
    """W warm-up and K timed steps of lmgc_encode (one model batch of the workload per step,
    inputs resident in HBM), CUDA events on the launching stream, max over ranks; per-class kernel
    times from the library's events inside the timed region; then, with e2e, the same K steps
    through lmgc_encode_host (pinned host buffers, copies inside the timed region)."""
    import numpy as np
    import torch
    import torch.distributed as dist

    tpv = L.lmgc_serial_tokens(ctx, vals.size) / vals.size  # tokens per value over the workload
    # values filling one model batch
    per_step = values_for_tokens(lambda m: L.lmgc_serial_tokens(ctx, m), vals.size, cfg.batch_windows * cfg.window)
    n_slices = max(1, vals.size // per_step)
    dev = torch.from_numpy(vals.view(np.int32) if vals.dtype == np.float32 else vals).cuda()
    slices = [dev[i * per_step:(i + 1) * per_step] for i in range(n_slices)]
    out = torch.empty(L.lmgc_encode_bound(ctx, per_step), dtype=torch.uint8, device="cuda")

    def step(k):
        return L.lmgc_encode(ctx, slices[(k + rank) % n_slices], out).numel()

    for k in range(args.warmup):
        step(k)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    L.lmgc_profile(ctx, True)
    l0 = L.lmgc_launch_count()
    sizes = []
    with Clocks(local) as clk:
        torch.cuda.synchronize()
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record()
        for k in range(args.steps):
            sizes.append(step(k))
        ev1.record()
        torch.cuda.synchronize()
    launches = L.lmgc_launch_count() - l0
    stats = L.lmgc_kernel_stats(ctx)
    L.lmgc_profile(ctx, False)
    ms = ev0.elapsed_time(ev1)
    if world > 1:
        t = torch.tensor([ms], device="cuda")
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
        dist.barrier()
    bpv = bytes_per_value(cfg)
    value = per_step * bpv * args.steps * world / (ms / 1e3) / 1e6
    del slices, dev

    e2e_res = None
    if e2e:  # end to end through host buffers
        src = vals.view(np.int32) if vals.dtype == np.float32 else vals
        hin = [torch.from_numpy(src[i * per_step:(i + 1) * per_step].copy()).pin_memory()
               for i in range(min(n_slices, 4))]
        hout = torch.empty(L.lmgc_encode_bound(ctx, per_step), dtype=torch.uint8).pin_memory()
        L.lmgc_encode_host(ctx, hin[0], hout)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        d2h = 0
        t0 = time.perf_counter()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for k in range(args.steps):
            d2h += L.lmgc_encode_host(ctx, hin[k % len(hin)], hout)
        e1.record()
        torch.cuda.synchronize()
        e2e_ms = e0.elapsed_time(e1)
        if world > 1:  # the slowest rank's time, as for the device-timed value
            t = torch.tensor([e2e_ms], device="cuda")
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            e2e_ms = float(t.item())
        e2e_res = {"value": per_step * bpv * args.steps * world / (e2e_ms / 1e3) / 1e6, "unit": "MB/s",
                   "h2d_bytes_per_step": per_step * bpv, "d2h_bytes_per_step": int(d2h / args.steps),
                   "wall_s": time.perf_counter() - t0}

    g = stats["gemm"]
    gemm_tflops = g["work"] / (g["ms"] / 1e3) / 1e12 if g["ms"] > 0 else 0.0
    traffic, traffic_src = profiled_traffic(name, "gemm_tc", g["work"] / max(1, g["launches"]))
    roofline = {"bound": "tensor", "kernel": "gemm (all linear layers and the vocabulary projection)",
                "achieved": gemm_tflops, "peak": pk["bf16_sus"], "unit": "TFLOP/s",
                "frac": gemm_tflops / pk["bf16_sus"],
                "peak_kind": f"bf16 sustained ({pk['src']}; fp16 MMAs run at the bf16 rate)",
                "launches": g["launches"], "avg_launch_ms": g["ms"] / max(1, g["launches"]),
                "algorithmic_flops_per_launch": g["work"] / max(1, g["launches"]),
                "traffic": traffic, "traffic_unit": "bytes per launch (DRAM read + write)",
                "traffic_source": traffic_src}
    stages = {}
    for cls, st in stats.items():
        if st["launches"] == 0:
            continue
        e = {"launches": st["launches"], "ms": st["ms"], "share": st["ms"] / ms if ms else None}
        if cls in ("gemm", "attention") and st["ms"] > 0:
            e.update(achieved=st["work"] / (st["ms"] / 1e3) / 1e12, unit="TFLOP/s")
            e["frac"] = e["achieved"] / pk["bf16_sus"]
        elif cls in ("cdf_pairs", "range_encode", "serialize") and st["ms"] > 0:
            e.update(achieved=st["work"] / (st["ms"] / 1e3) / 1e9, unit="GB/s")
            e["frac"] = e["achieved"] / pk["hbm"]
        stages[cls] = e
    return {"value": value, "ms": ms, "per_step": per_step, "tpv": tpv, "bpv": bpv, "clocks": clk.summary(),
            "launches": launches, "roofline": roofline, "stages": stages, "e2e": e2e_res,
            "stage_ms": L.lmgc_stage_times(ctx), "rate_pct": 100.0 * statistics.mean(sizes) / (per_step * bpv),
            "bits_per_token": 8.0 * statistics.mean(sizes) / L.lmgc_serial_tokens(ctx, per_step)}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=WORKLOADS)
    ap.add_argument("--batch-windows", type=int, default=0)
    # a model with fewer layers, for small profiler captures only (the config line names it)
    ap.add_argument("--layers", type=int, default=0)
    ap.add_argument("--ref-positions", type=int, default=12)
    ap.add_argument("--cpu-target-s", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-micro", action="store_true")
    # encode the whole workload once (every window, in batches of --batch-windows), then decode
    # the first, middle and last windows and check them; prints one JSON line of its own
    ap.add_argument("--full", action="store_true")
    # only the serialise and coder microbenchmarks (one JSON line), the coder on this many windows
    # of 2048 tokens (small profiler captures use 2^16)
    ap.add_argument("--micro-only", action="store_true")
    # decode throughput: encode one batch of windows, then time lmgc_decode of all of them
    # (KV-cached, one model step per position) and check the tokens; one JSON line of its own
    ap.add_argument("--decode", action="store_true")
    ap.add_argument("--decode-windows", type=int, default=0)  # windows to decode (default: one batch)
    ap.add_argument("--coder-windows", type=int, default=1 << 20)
    # the default workload's line also carries the TinyLlama-shaped step; this leaves it out
    ap.add_argument("--no-extra", action="store_true")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)

    import numpy as np
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")

    import __graft_entry__

    # one builder per node (the build writes in-tree files); the other ranks wait, then load
    if local == 0:
        __graft_entry__.build()
    if world > 1:
        dist.barrier()
    from paper_2409_17836_gb300 import configs, lmgc as L

    cfg, vals = workload(args.workload)
    if args.batch_windows:
        cfg = configs.with_(cfg, batch_windows=args.batch_windows)
    if args.layers:
        cfg = configs.with_(cfg, n_layers=args.layers)
    if args.micro_only:
        print(json.dumps({"mode": "micro", "microbench": micro_run(L, configs, peaks(), args.coder_windows)}),
              flush=True)
        return 0
    ctx = L.Context(cfg)
    if args.full:
        return run_full(args, cfg, ctx, vals)
    if args.decode:
        return run_decode(args, cfg, ctx, vals)
    pk = peaks()
    m = measure_steps(L, ctx, cfg, vals, args, world, rank, local, pk, args.workload)
    ctx.close()
    extra = None
    if args.workload == DEFAULT_WORKLOAD and not args.no_extra:
        # the TinyLlama-shaped step (2048-token windows, 64 per batch) beside the headline
        tcfg, tvals = workload("convnet-tinyllama")
        tctx = L.Context(tcfg)
        t = measure_steps(L, tctx, tcfg, tvals, args, world, rank, local, pk, "convnet-tinyllama", e2e=False)
        tctx.close()
        extra = {"workload": "convnet-tinyllama", "value": t["value"], "unit": "MB/s",
                 "ms_per_step": t["ms"] / args.steps, "model": model_name(tcfg), "window": tcfg.window,
                 "batch_windows": tcfg.batch_windows, "values_per_step": t["per_step"], "clocks": t["clocks"],
                 "roofline": t["roofline"], "stages": t["stages"], "gpu_launches": t["launches"]}
    ctx = None
    micro = None
    if rank == 0 and not args.no_micro and cfg.vocab == 32000:
        micro = micro_run(L, configs, pk, args.coder_windows)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(cfg, vals, m["tpv"], m["bpv"], args.cpu_target_s)
    if rank == 0:
        res = {"metric": METRIC, "value": m["value"], "unit": "MB/s", "n_gpus": world, "steps": args.steps,
               "warmup": args.warmup, "ms_per_step": m["ms"] / args.steps, "higher_is_better": True,
               "scaling": "weak", "vs_baseline": None, "dtype": "f16" if cfg.dtype == L.BF16 else "f32",
               "data": "synthetic (seeded random-init ConvNet gradients on Gaussian inputs; random-init model)",
               "config": {"workload": args.workload, "values_per_step": m["per_step"], "window": cfg.window,
                          "batch_windows": cfg.batch_windows, "cdf_bits": cfg.cdf_bits, "model": model_name(cfg),
                          "weights": "bf16 values (random init), held in fp16; fp16 activations, fp32 accumulation"
                          if cfg.dtype == L.BF16 else "fp32",
                          "l2": "no flush: each step reads > L2 (model weights and per-batch logits)",
                          "parallelism": f"windows sharded over {world} GPU(s), no collective on the data path"},
               "clocks": m["clocks"], "e2e": m["e2e"], "gpu_launches": m["launches"], "roofline": m["roofline"],
               "stages": m["stages"], "microbench": micro, "stage_ms_last_step": m["stage_ms"],
               "compression_rate_pct": m["rate_pct"], "bits_per_token": m["bits_per_token"],
               "cpu_baseline": cpu}
        if extra is not None:
            res["tinyllama_step"] = extra
        print(json.dumps(res), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()

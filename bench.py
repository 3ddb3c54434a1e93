"""Throughput benchmark of the AECCT batched decoder on GB300.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl {cuda,reference}] [--workload KEY]
                  [--variant {aecct,ecct,fp-hpsa}]

A step decodes one batch of the workload (default: BCH(63,36), d = 128, N = 10, 8 heads,
B = 262,144 received words, BPSK/AWGN at Eb/N0 cycling over 4, 5, 6, 7 dB: the largest
configuration, 92.8 T int ops per batch) through the C ABI (aecct_decode).  Inputs are resident in HBM before the timed region; L2 is flushed between
steps by writing a 256 MB buffer outside the timed events.  One JSON line is printed by
rank 0.  Under torchrun each rank decodes its own batch (weak scaling, no collective on the
data path); the time is the maximum over ranks.

--variant selects the model: aecct (default, the paper's method), ecct (the ECCT baseline of
Sec. 3: full-precision linears on bf16 tensor cores, the code-aware mask on every head, GELU) or
fp-hpsa (full-precision linears with HPSA and ReLU).

--impl reference times the CPU oracle (the plain C forward pass) on a bounded sample of
the same workload on the host cores, and reports the same metric.
"""
from __future__ import annotations

import argparse
import glob
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2410_05911_gb300 import inputs as I  # noqa: E402

METRIC = "decoded codewords/s"
UNIT = "codewords/s"


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm_gbs=p["hbm_gbs"], bf16_tflops=p["bf16_tflops"],
                    bf16_tflops_sustained=p.get("bf16_tflops_sustained", p["bf16_tflops"]), source="measured")
    return dict(hbm_gbs=6800.0, bf16_tflops=1900.0, bf16_tflops_sustained=1700.0, source="fallback")


def kernel_sources_digest() -> str:
    """SHA-256 over the CUDA sources and build flags of the decoder (paths and contents)."""
    h = hashlib.sha256()
    pkg = os.path.join(ROOT, "paper_2410_05911_gb300")
    files = sorted(glob.glob(os.path.join(pkg, "csrc", "*"))) + [os.path.join(pkg, "build_lib.py")]
    for f in files:
        if os.path.isfile(f) and f.endswith((".cu", ".cuh", ".h", ".py")):
            h.update(os.path.relpath(f, ROOT).encode())
            with open(f, "rb") as fh:
                h.update(fh.read())
    return h.hexdigest()


def measured_traffic(workload: str, batch: int):
    """DRAM bytes of one launch from the committed ncu record of this workload at this batch, or
    None when there is no record for it or the kernel sources changed since it was taken (the
    weights are read once per launch whatever the batch, so a record does not scale to another)."""
    path = os.path.join(ROOT, "profiles", f"aecct_decoder_kernel{I.WORKLOADS[workload]['d']}_{workload}_dram.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        rec = json.load(f)
    if rec.get("sources_sha256") != kernel_sources_digest() or rec.get("workload") != workload or rec.get("batch") != batch:
        return None
    return rec["dram_bytes_read"] + rec["dram_bytes_write"]


def max_over_ranks(x: float, world: int, device=None) -> float:
    """The maximum of x over the ranks of the process group (x itself when world == 1)."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist

    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def rank_seed(rank: int, i: int) -> int:
    """Seed of the i-th input batch of a rank: every rank decodes its own words (weak scaling)."""
    return 1000 * rank + 11 + i


def work_per_word(w: I.Workload):
    """Algorithmic work per decoded word: the paper's integer additions of the linear layers
    ((2n-k) d^2 per d x d layer, App. A) counted as 2 ops per multiply-accumulate, 12 d^2 per
    token per block; plus HBM bytes y in (4n), bits + syndrome out (n + n-k)."""
    T, d, N = w.code.T, w.d, w.n_layers
    return dict(int_ops=2 * 12 * T * d * d * N, io_bytes=4 * w.code.n + w.code.n + (w.code.n - w.code.k))


ALU_NOMINAL_TOPS = 152 * 128 * 2.070e9 / 1e12  # 152 SMs x 128 fp32 lanes x 2070 MHz (an FMA is one op), T ops/s


def measured_alu_peak():
    """The fp32 FMA rate measured on this device by the library's diagnostic kernel (scalar and
    paired f32x2 instructions; the larger), in T ops/s, an FMA counting one op."""
    from paper_2410_05911_gb300 import aecct

    rates = {"scalar": aecct.selftest_fma_rate(False) / 1e12, "paired": aecct.selftest_fma_rate(True) / 1e12}
    return max(rates.values()), rates


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the machine type)."""
    import platform

    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name"):
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


def alu_ops_per_word(code, model) -> float:
    """Algorithmic fp32 operations per decoded word of the canonical forward pass (an FMA, a
    compare-select or a divide is one op; the integer core on the tensor cores, integer index
    work and loads are not counted).  Per block and token, AAP linears with ReLU: Quant of a
    K-row 4K + 2 (max |x|, floor, 127/alpha, mul + two rounding adds per code), dequant of an
    N-row 2N + 2, residual + LayerNorm over d 8d + 3, ReLU 1 per hidden unit: 66d + 26 in all.
    HPSA per (token, head) with kappa keys: kappa (2 d_h + 16) + d_h + 1 (pass 1: d_h FMAs, the
    chain add, scale, max; pass 2: shift, 11 for exp2, the sum, d_h FMAs; then 1/l and d_h
    products).  Plus the embedding products and the output head."""
    H = code.H.astype(np.int64)
    m, n = H.shape
    T, d = n + m, model.d
    dh, heads = d // 8, 8
    F = model.ffn_mult * d
    deg_v, deg_c = H.sum(0), H.sum(1)
    m1 = np.concatenate([deg_v, deg_c])                       # first ring: Tanner neighbours
    vv = (H.T @ H) > 0
    cc = (H @ H.T) > 0
    m2 = np.concatenate([vv.sum(1), cc.sum(1)])               # second ring, with the node itself
    if getattr(model, "mask_mode", 0) == 1:
        keys = heads * (m1 + m2).sum()                         # the rings are disjoint: union size = sum
    else:
        keys = model.h_first * m1.sum() + (heads - model.h_first) * m2.sum()
    attn = keys * (2 * dh + 16) + T * heads * (dh + 1)
    act = 1 if model.activation == 0 else 25                   # GELU: its erf and exp2 steps
    if getattr(model, "linear_mode", 0) == 0:
        quant = lambda K: 4 * K + 2                            # noqa: E731
        deq = lambda N: 2 * N + 2                              # noqa: E731
    else:                                                      # bf16 rounding, acc + b
        quant = lambda K: K                                    # noqa: E731
        deq = lambda N: N                                      # noqa: E731
    ln = 8 * d + 3
    per_token = (quant(d) + deq(3 * d) + 4 + quant(d) + deq(d) + ln + quant(d) + deq(F) + act * F + quant(F)
                 + deq(d) + ln)
    per_layer = T * per_token + attn
    head = T * (d - model.d_spe) + T * (2 * d + 1) + n * (T + 1) + n
    return float(model.n_layers * per_layer + head)


class ClockSampler:
    """nvidia-smi clocks and throttle reasons during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-i", str(self.gpu), "-lms", "100"], stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if not self.lines:
            return None
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx = max(mx, float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return dict(sm_mhz=float(np.median(sm)), sm_max_mhz=mx, reasons=sorted(reasons), samples=len(sm))


def cpu_oracle_rate(model, y, budget_s: float = 12.0, chunk: int = 64, max_words: int = 8192, threads: int = 0):
    """Oracle decode rate (words/s) on the host cores over a bounded prefix of y; also returns the
    oracle's outputs for the words it decoded (the parity sample)."""
    from oracle import oracle as O

    cores = threads or os.cpu_count() or 1
    chunk = max(cores, chunk) if threads == 0 else chunk
    done, t0 = 0, time.perf_counter()
    outs = []
    while done < min(max_words, y.shape[0]):
        outs.append(O.decode(model, y[done:done + chunk], nthreads=cores))
        done += min(chunk, y.shape[0] - done)
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    ref = {k: np.concatenate([o[k] for o in outs]) for k in ("bits", "syndrome", "logits")}
    return done / dt, done, dt, cores, ref


def parity_summary(gpu: dict, ref: dict) -> dict:
    """GPU outputs against the oracle's on the same words: bit-exact logits and decisions, and
    the tolerance criteria (|d logit| <= 2e-2; decisions equal except where |logit| < 0.05)."""
    dl = np.abs(gpu["logits"].astype(np.float64) - ref["logits"].astype(np.float64))
    differ = gpu["bits"] != ref["bits"]
    return dict(words=int(ref["bits"].shape[0]), bits=int(ref["bits"].size),
                logits_bit_exact=bool((gpu["logits"].view(np.int32) == ref["logits"].view(np.int32)).all()),
                max_abs_dlogit=float(dl.max()), bits_differ=int(differ.sum()),
                bits_differ_away_from_zero=int((differ & (np.abs(ref["logits"]) >= 0.05)).sum()),
                syndromes_equal=bool((gpu["syndrome"] == ref["syndrome"]).all()))


VARIANTS = {
    # name: (model overrides, mask_mode, description)
    "aecct": (dict(), 0, "AECCT: AAP ternary linears, HPSA, ReLU"),
    "ecct": (dict(full_precision=True, activation=1), 1,
             "ECCT baseline: full-precision (bf16) linears, code-aware mask on every head, GELU"),
    "fp-hpsa": (dict(full_precision=True), 0, "full-precision (bf16) linears with HPSA and ReLU"),
}


def variant_model(key: str, variant: str):
    overrides, mask_mode, _ = VARIANTS[variant]
    model = I.workload_model(key, **overrides)
    model.mask_mode = mask_mode
    return model


def run_reference(args, rank, world):
    w = I.workload(args.workload)
    model = variant_model(args.workload, args.variant)
    if rank != 0:
        return
    chunk = max(16, w.code.T and 64)
    ys = [I.channel_batch(w.code, 1024, e, seed=7 + i).y for i, e in enumerate(w.ebn0_db)]
    per_step_budget = max(1.0, 60.0 / max(1, args.steps + args.warmup))
    from oracle import oracle as O

    cores = os.cpu_count() or 1
    for s in range(args.warmup):
        O.decode(model, ys[s % len(ys)][:16], nthreads=cores)
    words, secs = 0, 0.0
    for s in range(args.steps):
        y = ys[s % len(ys)]
        t0 = time.perf_counter()
        done = 0
        while done < y.shape[0]:
            O.decode(model, y[done:done + chunk], nthreads=cores)
            done += chunk
            if time.perf_counter() - t0 > per_step_budget:
                break
        secs += time.perf_counter() - t0
        words += done
    value = words / secs
    line = dict(metric=METRIC, value=value, unit=UNIT, n_gpus=world, steps=args.steps, warmup=args.warmup,
                ms_per_step=1e3 * secs / args.steps, higher_is_better=True, scaling="weak", vs_baseline=None,
                dtype="i8/f32" if args.variant == "aecct" else "bf16/f32", data="synthetic", impl="reference",
                config=dict(workload=workload_label(w), batch=w.batch, variant=args.variant),
                cpu_baseline=dict(value=value, unit=UNIT, cores=cores, kind="oracle",
                                  sample=f"{words} words over {args.steps} steps, each a time-bounded prefix of a "
                                         f"1024-word batch of the workload"),
                e2e=dict(value=value, unit=UNIT, h2d_bytes_per_step=0, d2h_bytes_per_step=0))
    print(json.dumps(line), flush=True)


def workload_label(w: I.Workload) -> str:
    return (f"{w.code.name} d={w.d} N={w.n_layers} heads=8 (4 first-ring/4 second-ring) T={w.code.T} "
            f"B={w.batch} Eb/N0={'/'.join(str(e) for e in w.ebn0_db)} dB")


def run_cuda(args, rank, world, local_rank):
    import torch

    from paper_2410_05911_gb300 import aecct

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = I.workload(args.workload)
    model = variant_model(args.workload, args.variant)
    B = args.batch or w.batch
    dec = aecct.Decoder(model)
    q = dec.query()
    # inputs: one batch per Eb/N0 point, resident on the device
    ys_host = [I.channel_batch(w.code, B, e, seed=rank_seed(rank, i)).y for i, e in enumerate(w.ebn0_db)]
    ys = [torch.from_numpy(y).to(dev) for y in ys_host]
    bits = torch.empty((B, w.code.n), dtype=torch.uint8, device=dev)
    syn = torch.empty((B, w.code.n - w.code.k), dtype=torch.uint8, device=dev)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step(i):
        dec.decode(ys[i % len(ys)], out=(bits, syn, None), stream=stream)

    # the CUDA-core roofline's denominator, measured before the timed region
    alu_peak, alu_rates = measured_alu_peak() if rank == 0 else (ALU_NOMINAL_TOPS, {})

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    if dec.synchronize() != aecct.AECCT_OK:
        raise RuntimeError("warm-up decode failed")
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    with ClockSampler(local_rank) as clk:
        time.sleep(0.3)
        if args.back_to_back:
            # the steps as one back-to-back sequence of launches between two events (L2 warm;
            # for batches whose launch is short enough for per-launch gaps to matter)
            flush.fill_(0.0)
            evs[0][0].record(stream)
            for i in range(args.steps):
                step(i)
            evs[0][1].record(stream)
        else:
            for i in range(args.steps):
                flush.fill_(float(i))
                evs[i][0].record(stream)
                step(i)
                evs[i][1].record(stream)
        torch.cuda.synchronize()
        time.sleep(0.2)
    if world > 1:
        dist.barrier()
    if dec.synchronize() != aecct.AECCT_OK:
        raise RuntimeError("timed decode reported an error")
    ms = [evs[0][0].elapsed_time(evs[0][1])] if args.back_to_back else [a.elapsed_time(b) for a, b in evs]
    total_s = max_over_ranks(sum(ms) / 1e3, world, dev)
    value = world * B * args.steps / total_s
    kernel_s = total_s / args.steps

    # end to end through the public host-buffer entry point: pinned y in, bits + syndrome out
    y_pin = torch.from_numpy(ys_host[0]).pin_memory()
    e2e_steps = max(3, min(args.steps, 20))
    dec.decode_host(y_pin.numpy(), want_logits=False)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for i in range(e2e_steps):
        dec.decode_host(y_pin.numpy(), want_logits=False)
    e2e_s = max_over_ranks((time.perf_counter() - t0) / e2e_steps, world, dev)
    e2e = dict(value=world * B / e2e_s, unit=UNIT, h2d_bytes_per_step=4 * B * w.code.n,
               d2h_bytes_per_step=B * w.code.n + B * (w.code.n - w.code.k))

    if rank != 0:
        return
    pk = peaks()
    wk = work_per_word(w)
    achieved_tops = wk["int_ops"] * B / kernel_s / 1e12
    tensor = dict(bound="tensor", achieved=achieved_tops, peak=pk["bf16_tflops"], unit="TFLOP/s",
                  frac=achieved_tops / pk["bf16_tflops"],
                  work="2*12*T*d^2*N ops per word on the bf16 tensor cores (AAP: exact integers; "
                       "full-precision linears: bf16 products); peak = measured bf16 dense burst")
    alu_tops = alu_ops_per_word(w.code, model) * B / kernel_s / 1e12
    alu = dict(bound="alu", achieved=alu_tops, peak=alu_peak, unit="TFLOP/s", frac=alu_tops / alu_peak,
               work="algorithmic fp32 ops of the canonical forward pass per word (bench.alu_ops_per_word; an FMA "
                    "is one op); peak = fp32 FMA rate measured on this GPU by aecct_selftest_fma_rate (the larger "
                    f"of scalar {alu_rates['scalar']:.1f} and paired {alu_rates['paired']:.1f} T FMA/s; nominal "
                    f"152 SMs x 128 lanes x 2070 MHz = {ALU_NOMINAL_TOPS:.1f})")
    # d <= 64: the fp32 work (HPSA, epilogues) binds; d = 128: the linear layers' contraction
    roof = dict(alu if w.d <= 64 else tensor)
    roof.update(traffic=args.traffic if args.traffic is not None else
                (measured_traffic(args.workload, B) if args.variant == "aecct" else None),
                kernel=f"aecct_decoder_kernel<{w.d}, {int(q['attention_mode'] == 2)}, {model.activation}, "
                       f"{model.linear_mode}>",
                other={k: v for k, v in (("tensor", tensor), ("alu", alu)) if v["bound"] != roof["bound"]})
    cpu = None
    parity = None
    if not args.no_cpu_baseline:
        rate, words, secs, cores, ref = cpu_oracle_rate(model, ys_host[0], budget_s=args.cpu_budget)
        rate1, words1, secs1, _, _ = cpu_oracle_rate(model, ys_host[0], budget_s=args.cpu_budget / 3, chunk=4,
                                                      threads=1)
        cpu = dict(value=rate, unit=UNIT, cores=cores, kind="oracle", cpu_model=cpu_model(),
                   sample=f"first {words} words of the {w.ebn0_db[0]} dB batch ({secs:.1f} s, {cores} threads)",
                   one_thread=dict(value=rate1, unit=UNIT, sample=f"first {words1} words ({secs1:.1f} s)"))
        # the GPU's outputs on the oracle's sample, compared with the oracle's
        g_bits, g_syn, g_logits = dec.decode(ys[0][:words])
        torch.cuda.synchronize()
        if dec.synchronize() != aecct.AECCT_OK:
            raise RuntimeError("parity decode reported an error")
        parity = parity_summary(dict(bits=g_bits.cpu().numpy(), syndrome=g_syn.cpu().numpy(),
                                     logits=g_logits.cpu().numpy()), ref)
    line = dict(
        metric=METRIC, value=value, unit=UNIT, n_gpus=world, steps=args.steps, warmup=args.warmup,
        ms_per_step=1e3 * kernel_s, higher_is_better=True, scaling="weak", vs_baseline=None,
        dtype="i8/f32" if args.variant == "aecct" else "bf16/f32", data="synthetic",
        config=dict(workload=workload_label(w), variant=args.variant, batch=B, tokens=w.code.T,
                    cluster_ctas=q["cluster_ctas"],
                    words_per_group=q["words_per_group"],
                    l2=("not flushed: the steps timed back to back as one sequence" if args.back_to_back
                        else "flushed between steps (256 MB write)"),
                    info_gbit_s=value * w.code.k / 1e9, hbm_io_gbs=value * wk["io_bytes"] / 1e9),
        e2e=e2e, roofline=roof, cpu_baseline=cpu, parity=parity, gpu_launches=args.steps, clocks=clk.summary())
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="cuda", choices=["cuda", "reference"])
    ap.add_argument("--workload", default="bch63_36", choices=sorted(I.WORKLOADS))
    ap.add_argument("--batch", type=int, default=0, help="override the batch size (0 = the workload's)")
    ap.add_argument("--variant", default="aecct", choices=sorted(VARIANTS),
                    help="; ".join(f"{k}: {v[2]}" for k, v in VARIANTS.items()))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--traffic", type=float, default=None, help="ncu DRAM bytes per launch, if measured")
    ap.add_argument("--back-to-back", action="store_true",
                    help="time the steps as one back-to-back sequence of launches without the L2 flush between them")
    args = ap.parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist

        backend = "nccl" if args.impl == "cuda" else "gloo"
        if backend == "nccl":
            import torch
            torch.cuda.set_device(local_rank)
        dist.init_process_group(backend=backend)
    try:
        if args.impl == "reference":
            run_reference(args, rank, world)
        else:
            run_cuda(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()

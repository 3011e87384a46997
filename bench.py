"""Benchmark of the FrameFT adapter hot path: fused forward + dX + dC over every
adapted matrix of the LLaMA-2-7B-shaped workload (32 layers x q/k/v/o,
4096 x 4096, 4096-entry shared support, 8192 bf16 tokens), one step = one
pass of the whole path over one batch.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Prints one JSON line (rank 0).  Under torchrun every rank runs its own
replica of the workload (the path needs no exchange between GPUs; weak
scaling) and the timing is the max over ranks.  Besides the headline, the
line carries ``per_config``: the same fused step timed on each of the five
evaluation workloads and the 64-tenant merge, each against its algorithmic
bytes, with the fp64 oracle sampled beside it.
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

METRIC = "adapter fwd+bwd tokens/sec at LLaMA-7B shape; achieved HBM GB/s vs 8 TB/s"
NOMINAL_GBS = 8000.0
L2_BYTES = 126 * 1024 * 1024

# evaluation workloads reported in per_config, in the order of their configs,
# then the paper's own rho = 2 regime at the LLaMA-2 shape (the dense path)
PER_CONFIG = ("single_256_fp32", "roberta_base_qv", "llama2_7b_qkvo", "llama3_8b_all", "vit_b16_merge",
              "llama2_rho2")


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="framefb", choices=["framefb", "reference"])
    p.add_argument("--workload", default=None)
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu", action="store_true")
    p.add_argument("--no-optimizer", action="store_true", help="skip the timing of the AdamW step")
    p.add_argument("--no-per-config", action="store_true", help="skip the per-config timings")
    p.add_argument("--configs", default=",".join(PER_CONFIG), help="comma-separated workloads for per_config")
    p.add_argument("--serving", action="store_true",
                   help="also time the mixed-tenant forward on ViT-B/16 shapes (64 images, one tenant each)")
    p.add_argument("--cpu-tokens", type=int, default=8192, help="token sample of the CPU oracle baseline")
    p.add_argument("--cpu-mats", type=int, default=4, help="matrices in the CPU oracle baseline sample")
    p.add_argument("--mats", type=int, default=None, help="first MATS matrices only (small profiling cases)")
    p.add_argument("--tokens", type=int, default=None, help="tokens per matrix (small profiling cases)")
    p.add_argument("--merge-only", action="store_true", help="time only the 64-tenant ViT-B/16 merge")
    return p.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def tensor_peak():
    """Sustained bf16 tensor peak (TFLOP/s) for kernels timed inside a long step."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 1700.0, "fallback"


def dense_flops(batch) -> float:
    """Algorithmic flops of one fused step on the dense path: the four dense
    contractions X Phi_in, dY Phi_out, Z Phi_out^T and G Phi_in^T, each
    2 N d K (K = k*rho frame columns); the SpMM's 6 N nnz is added."""
    total = 0.0
    for b in batch.bufs:
        fin, fout = batch.frames[b.spec.n], batch.frames[b.spec.m]
        total += 4.0 * batch.N * (b.spec.n * fin.ncols + b.spec.m * fout.ncols) + 6.0 * batch.N * batch.w.nnz
    return total


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
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
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def _read(self):
        for ln in self.proc.stdout:
            self.lines.append(ln.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
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
            for nm, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def algorithmic_bytes(batch) -> int:
    """Minimum HBM bytes of one fused step: X and dY read once, Y and dX
    read-modify-written, over the coordinates of groups the support touches,
    plus C values, dC and 8 bytes of indices per support entry."""
    import numpy as np
    total = 0
    esz = 2 if batch.w.dtype == "bf16" else 4
    for b, key in zip(batch.bufs, batch.keys):
        img = batch.plans[key].image()
        hdr = np.frombuffer(img[:128].tobytes(), dtype=np.int32)
        Gn, Gm, nnz = int(hdr[4]), int(hdr[5]), int(hdr[6])
        zmask = np.frombuffer(img[hdr[21]:hdr[21] + 4 * Gm].tobytes(), dtype=np.uint32)
        gmask = np.frombuffer(img[hdr[22]:hdr[22] + 4 * Gn].tobytes(), dtype=np.uint32)
        r_out, r_in = 32 * int(np.count_nonzero(zmask)), 32 * int(np.count_nonzero(gmask))
        if int(hdr[26]) == 1:  # dense path: Phi touches every coordinate
            r_out, r_in = b.spec.m, b.spec.n
        total += 3 * esz * batch.N * (r_in + r_out) + nnz * (4 + 4 + 8)
    return total


def merge_bytes(m: int, n: int, T: int, nnz: int, esz: int) -> int:
    """Minimum HBM bytes of a T-tenant merge: W0 read once, every W_t written,
    the tenants' C values and the support indices read."""
    return esz * m * n * (T + 1) + T * nnz * 4 + nnz * 8


# sources of the dominant kernel (bf16: the two-token tcgen05 kernel unless
# FRAMEFB_KERNEL selects another) and of the plan builder that shapes it
KERNEL_SOURCES = ("framefb_kernels.cuh", "framefb_mma.cuh", "framefb_ptx.cuh", "framefb_tc.cuh", "framefb_tc2.cuh",
                  "plan_layout.h", "framefb_host.cpp")


def kernel_choice():
    k = os.environ.get("FRAMEFB_KERNEL", "tc2")
    return k if k in ("tile", "tc") else "tc2"


def measured_traffic():
    """ncu DRAM bytes per launch of the dominant kernel, if taken on the current
    kernel sources with the same kernel choice."""
    import hashlib
    try:
        csrc = os.path.join(ROOT, "paper_2608_26430_gb300", "csrc")
        hh = hashlib.sha256()
        for name in KERNEL_SOURCES:
            hh.update(open(os.path.join(csrc, name), "rb").read())
        h = hh.hexdigest()[:16]
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            rec = json.load(f).get(h, {})
        if rec.get("kernel_choice") != kernel_choice():
            return None
        return rec.get("bytes_per_launch")
    except Exception:
        return None


# ---------------------------------------------------------------------------
# CPU side: the oracle as it stands, and what the host is
# ---------------------------------------------------------------------------
def cpu_threads():
    try:
        from threadpoolctl import threadpool_info
        info = threadpool_info()
        if info:
            return max(int(i.get("num_threads", 1)) for i in info)
    except Exception:
        pass
    return os.cpu_count() or 1


def cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.strip().lower().startswith("model name"):
                return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    return "unknown"


def host_info() -> dict:
    return {"nproc": os.cpu_count(), "cpu_model": cpu_model(), "blas_threads": cpu_threads()}


def oracle_flops(m: int, n: int, N: int) -> float:
    """Dense fp64 flops of the oracle for one matrix over N tokens (k*rho = d
    frames, so K_m = m and K_n = n): dW = P_m C P_n^T twice (forward and dX),
    X dW^T, dY dW, and dY^T X followed by P_m^T (.) P_n for dC."""
    dw = 2.0 * (m * m * n + m * n * n)
    return 2 * dw + 2.0 * N * m * n * 3 + dw


def cpu_oracle_sample(w, tokens: int, mats=(0,)):
    """Time the oracle (fp64 numpy) on the given matrices of the workload over
    `tokens` tokens each; returns (compute seconds, setup seconds)."""
    import numpy as np
    from oracle import adapter, frames, support
    from paper_2608_26430_gb300 import workloads as wl
    tcomp = tsetup = 0.0
    for j in mats:
        spec = w.mats[j]
        X = wl.x_input(w, j, tokens).float().numpy().astype(np.float64)
        dY = wl.dy_input(w, j, tokens).float().numpy().astype(np.float64)
        c = wl.c_values(w, j).numpy().astype(np.float64)
        s = wl.scale_of(w, spec)
        t0 = time.perf_counter()
        Pin = frames.real_frame(spec.n, w.k, spec.n // w.k)
        Pout = Pin if spec.m == spec.n else frames.real_frame(spec.m, w.k, spec.m // w.k)
        row, col, _, _ = support.sample_support(spec.m, spec.n, w.nnz, wl.support_seed_of(w, j), w.support_mode,
                                                w.zipf_s, w.k)
        t1 = time.perf_counter()
        C = adapter.dense_C(spec.m, spec.n, row, col, c)
        adapter.forward(X, np.zeros((tokens, spec.m)), Pin, Pout, C, s)
        adapter.backward_dx(dY, np.zeros((tokens, spec.n)), Pin, Pout, C, s)
        adapter.grad_coeff(X, dY, Pin, Pout, s, row, col)
        t2 = time.perf_counter()
        tcomp += t2 - t1
        tsetup += t1 - t0
    return tcomp, tsetup


def oracle_step_estimate(w, tokens: int, mats=(0,)):
    """The oracle timed on a sample (the given matrices over `tokens` tokens),
    scaled to a full step of the workload by the dense oracle's flop count:
    returns (tokens/s, sample seconds, sample description)."""
    t, _ = cpu_oracle_sample(w, tokens, mats)
    f_sample = sum(oracle_flops(w.mats[j].m, w.mats[j].n, tokens) for j in mats)
    f_step = sum(oracle_flops(s.m, s.n, w.N) for s in w.mats)
    step_s = t * f_step / f_sample
    shapes = ", ".join(f"{w.mats[j].m}x{w.mats[j].n}" for j in mats)
    desc = (f"dense fp64 oracle on {len(mats)} of {len(w.mats)} matrices ({shapes}) over {tokens} of {w.N} tokens "
            f"({t:.2f} s), scaled to the full step by the oracle's flop count")
    return w.N / step_s, t, desc


def config_of(w, nmats: int, world: int) -> dict:
    """The workload description both arms print.  The timed steps do not flush
    L2: the bytes of X, dY, Y and dX one step touches say whether they can stay
    in it (the full evaluation workloads: no; the small profiling cases: yes)."""
    esz = 4 if w.dtype == "f32" else 2
    touched = 2 * esz * w.N * sum(s.n + s.m for s in w.mats[:nmats])
    l2 = (f"inputs larger than L2 ({touched / 2 ** 30:.0f} GiB of X, dY, Y and dX per step)" if touched > 2 * L2_BYTES
          else f"{touched / 2 ** 20:.0f} MiB of X, dY, Y and dX per step, L2 not flushed (a profiling case)")
    return {"workload": w.name, "matrices": nmats, "tokens": w.N, "nnz": w.nnz,
            "shape": f"{w.mats[0].m}x{w.mats[0].n}", "k": w.k, "parallelism": "replicas" if world > 1 else "single",
            "l2": l2}


def max_over_ranks(ms: float, world: int, device) -> float:
    """The slowest rank's time (every rank's timed region counts)."""
    import torch
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def reference_arm(args, w, rank, world):
    """The oracle as it stands on the host cores (the paper ships no code):
    each step is one matrix of the workload over cpu_tokens tokens, scaled to
    the full step."""
    if rank != 0:
        return
    per = []
    for i in range(args.warmup + args.steps):
        t, _ = cpu_oracle_sample(w, args.cpu_tokens)
        if i >= args.warmup:
            per.append(t)
    step = sum(per) / len(per)
    # the sample is one of the workload's matrices over cpu_tokens tokens; the
    # full step is len(mats) matrices over N tokens
    tok_s = args.cpu_tokens / (step * len(w.mats))
    out = {"impl": "reference", "metric": METRIC, "value": tok_s, "unit": "tokens/s", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": step * 1e3 * len(w.mats) * w.N / args.cpu_tokens,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": config_of(w, len(w.mats), world),
           "cpu_baseline": {"value": tok_s, "unit": "tokens/s", "cores": cpu_threads(), "kind": "oracle",
                            "sample": f"dense fp64 oracle, 1 of {len(w.mats)} matrices ({w.mats[0].m}x{w.mats[0].n}), "
                                      f"{args.cpu_tokens} of {w.N} tokens per step, scaled to the full step",
                            **host_info()},
           "e2e": {"value": tok_s, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


# ---------------------------------------------------------------------------
# GPU side
# ---------------------------------------------------------------------------
class L2Flush:
    """Writes a buffer larger than L2 between timed iterations."""

    def __init__(self, dev):
        import torch
        self.buf = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=dev)

    def __call__(self):
        self.buf.fill_(1.0)


def time_steps(fn, stream, steps: int, warmup: int, flush=None):
    """Mean CUDA-event time (ms) of `fn` over `steps` calls on `stream`, each
    call timed on its own; `flush` (outside the events) runs before each."""
    import torch
    for _ in range(warmup):
        if flush:
            flush()
        fn()
    torch.cuda.synchronize()
    ms = []
    for _ in range(steps):
        if flush:
            flush()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        ms.append((a, b))
    torch.cuda.synchronize()
    return statistics.mean(a.elapsed_time(b) for a, b in ms)


def time_config(name, dev, stream, steps, warmup, flush, with_cpu, headline=None):
    """One fused fwd + dX + dC step over every matrix of workload `name`."""
    import torch
    from paper_2608_26430_gb300 import framefb as ffb
    from paper_2608_26430_gb300 import workloads as wl
    from paper_2608_26430_gb300.batch import AdapterBatch
    w = wl.WORKLOADS[name]
    ops = ffb.OP_FORWARD | ffb.OP_BACKWARD_DX | ffb.OP_GRAD_COEFF
    peak, _ = peaks()
    flops = None
    if headline is not None:
        ms, alg, kernels = headline
    else:
        batch = AdapterBatch(w, dev, ops=ops)
        ws = batch.workspace(ops)
        alg = algorithmic_bytes(batch)
        if not all(f.structured for f in batch.frames.values()):
            flops = dense_flops(batch)
        kernels = ffb.framefb_kernel_names(batch.mats, ops, batch.dtype_code)
        small = alg < 2 * L2_BYTES
        ms = time_steps(lambda: batch.run(ops, ws, stream), stream, steps, warmup, flush if small else None)
        del batch, ws
        torch.cuda.empty_cache()
    gbs = alg / (ms / 1e3) / 1e9
    rec = {"ms_per_step": ms, "tokens_per_s": w.N / (ms / 1e3), "matrices": len(w.mats), "tokens": w.N,
           "dtype": w.dtype, "algorithmic_bytes": alg, "achieved_gbs": gbs, "frac_of_measured": gbs / peak,
           "frac_of_8tbs": gbs / NOMINAL_GBS,
           "kernels": kernels + ([] if any(k.startswith("dense") for k in kernels) else ["dc_reduce_kernel"]),
           "l2": "L2 flushed between steps" if alg < 2 * L2_BYTES else "step moves more than L2"}
    if flops:
        tpk, kind = tensor_peak()
        tf = flops / (ms / 1e3) / 1e12
        # each algorithmic flop costs two bf16 tensor-core flops on this path:
        # the analysis multiplies by Phi split into bf16 hi + lo parts, the
        # synthesis runs at the tf32 rate (half the bf16 rate)
        rec["roofline"] = {"bound": "tensor", "algorithmic_flops": flops, "achieved_tflops": tf,
                           "peak_tflops": tpk / 2, "frac": tf / (tpk / 2),
                           "peak": f"bf16 sustained ({kind}) / 2: two bf16 tensor flops per algorithmic flop"}
    if with_cpu:
        shapes = []
        for j, s in enumerate(w.mats):
            if (s.m, s.n) not in [(w.mats[i].m, w.mats[i].n) for i in shapes]:
                shapes.append(j)
        # fp64 BLAS on the largest shapes takes minutes per matrix: the sample
        # keeps the shapes up to 4096 and fewer tokens for the large workloads
        big = max(max(w.mats[j].m, w.mats[j].n) for j in shapes)
        tokens = min(w.N, 2048 if big <= 4096 else 512)
        shapes = [j for j in shapes if max(w.mats[j].m, w.mats[j].n) <= 4096]
        tok_s, t, desc = oracle_step_estimate(w, tokens, tuple(shapes))
        rec["cpu_oracle"] = {"value": tok_s, "unit": "tokens/s", "sample_s": t, "sample": desc,
                             "cores": cpu_threads()}
    return rec


def time_merge(dev, stream, steps, warmup, flush):
    """The 64-tenant merge of the ViT-B/16 workload (768 x 768 bf16 W0)."""
    import torch
    from paper_2608_26430_gb300 import framefb as ffb
    from paper_2608_26430_gb300 import workloads as wl
    w = wl.WORKLOADS["vit_b16_merge"]
    m, n = w.merge_shape
    T = w.merge_tenants
    fin, fout = ffb.Frame(n, w.k, n // w.k), ffb.Frame(m, w.k, m // w.k)
    row, col, _, _ = ffb.framefb_support_build(m, n, w.nnz, w.support_seed, w.support_mode, w.zipf_s, w.k)
    plan = ffb.Plan(fin, fout, row, col)
    pd, dfin, dfout = plan.to_device(dev), fin.to_device(dev), fout.to_device(dev)
    W0 = wl.w0_input(w, dev)
    cv = wl.merge_c_values(w, dev)
    Wout = torch.empty((T, m, n), device=dev, dtype=W0.dtype)
    s = w.alpha / (m * n) ** 0.5
    ms = time_steps(lambda: ffb.framefb_merge(W0, dfin, dfout, plan, pd, cv, T, s, Wout, stream), stream,
                    steps, warmup, flush)
    nb = merge_bytes(m, n, T, w.nnz, 2)
    peak, _ = peaks()
    gbs = nb / (ms / 1e3) / 1e9
    return {"ms_per_call": ms, "tenants": T, "shape": f"{m}x{n}", "dtype": "bf16", "algorithmic_bytes": nb,
            "achieved_gbs": gbs, "frac_of_measured": gbs / peak, "frac_of_8tbs": gbs / NOMINAL_GBS,
            "kernels": ["merge_kernel<bf16>"], "l2": "L2 flushed between calls"}


def serving_timing(dev, stream, reps: int = 10):
    """Forward-only ViT-B/16 step (72 matrices, 64 images x 197 tokens) with
    one tenant per image through framefb_forward_tenants (the segment table
    in the kernel's launch parameters, and, for comparison, one launch
    matrix per (matrix, segment) with FRAMEFB_SEG_KERNEL=0), against the
    same step with one tenant for all tokens (framefb_forward)."""
    import torch
    from paper_2608_26430_gb300 import framefb as ffb
    from paper_2608_26430_gb300 import workloads as wl
    from paper_2608_26430_gb300.batch import AdapterBatch
    w = wl.WORKLOADS["vit_b16_merge"]
    T, per = 64, 197
    b = AdapterBatch(w, dev, ops=ffb.OP_FORWARD)
    cv = [wl.normal((T, w.nnz), 900 + i, w.c_std, device=dev) for i in range(len(b.mats))]
    mats = []
    for mat, c in zip(b.mats, cv):
        m2 = ffb.framefb_mat.from_buffer_copy(mat)
        m2.c_val = c.data_ptr()
        mats.append(m2)
    starts, tenants = [per * i for i in range(T + 1)], list(range(T))

    def timed(fn):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            fn()
        z.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(z) / reps

    ms_t = timed(lambda: ffb.framefb_forward_tenants(mats, b.dtype_code, starts, tenants, T, stream))
    os.environ["FRAMEFB_SEG_KERNEL"] = "0"
    try:
        ms_s = timed(lambda: ffb.framefb_forward_tenants(mats, b.dtype_code, starts, tenants, T, stream))
    finally:
        del os.environ["FRAMEFB_SEG_KERNEL"]
    ms_1 = timed(lambda: ffb.framefb_forward(b.mats, b.dtype_code, None, stream))
    return {"workload": "vit_b16 forward, 72 matrices, 64 images x 197 tokens", "tenants": T,
            "ms_mixed_tenants": ms_t, "ms_one_tenant": ms_1, "mixed_over_one_tenant": ms_t / ms_1,
            "ms_mixed_per_segment_launches": ms_s, "tokens_per_s_mixed": w.N / (ms_t / 1e3),
            "tokens_per_s_one_tenant": w.N / (ms_1 / 1e3), "l2": "step moves more than L2"}


def e2e_timing(batch, ops, ws, stream, steps, world, dev, barrier):
    """The same step through the same C-ABI call with host buffers: per step
    X, dY, Y and dX (Y and dX are read-modify-written) are copied in from
    pinned host memory and Y, dX and dC read back."""
    import torch
    w = batch.w
    hin = []
    for b in batch.bufs:
        for t in (b.X, b.dY, b.Y, b.dX):
            hin.append((torch.empty(t.shape, dtype=t.dtype, pin_memory=True), t))
    for h, t in hin:
        h.copy_(t)
    hout = []
    for b in batch.bufs:
        for t in (b.Y, b.dX, b.dC):
            hout.append((torch.empty(t.shape, dtype=t.dtype, pin_memory=True), t))
    h2d = sum(h.numel() * h.element_size() for h, _ in hin)
    d2h = sum(h.numel() * h.element_size() for h, _ in hout)

    def step():
        for h, t in hin:
            t.copy_(h, non_blocking=True)
        batch.run(ops, ws, stream)
        for h, t in hout:
            h.copy_(t, non_blocking=True)
    step()
    torch.cuda.synchronize()
    barrier()
    s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s0.record(stream)
    for _ in range(steps):
        step()
    s1.record(stream)
    torch.cuda.synchronize()
    te = max_over_ranks(s0.elapsed_time(s1) / steps, world, dev)
    del hin, hout
    return {"value": w.N * world / (te / 1e3), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": steps,
            "moves": "X, dY, Y, dX host to device; Y, dX, dC device to host"}


def main():
    args = parse()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    from paper_2608_26430_gb300 import workloads as wl
    w = wl.WORKLOADS[args.workload or wl.HEADLINE]
    if args.tokens is not None:
        import dataclasses
        w = dataclasses.replace(w, N=args.tokens)
    if args.impl == "reference":
        return reference_arm(args, w, rank, world)

    import torch
    import torch.distributed as dist
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device(dev))

    def barrier():
        if world > 1:
            dist.barrier()

    from __graft_entry__ import build
    build()
    from paper_2608_26430_gb300 import framefb as ffb
    from paper_2608_26430_gb300.batch import AdapterBatch

    if args.merge_only:
        rec = time_merge(dev, torch.cuda.current_stream(), args.steps, args.warmup, L2Flush(dev))
        if rank == 0:
            print(json.dumps({"merge": rec}), flush=True)
        return

    ops = ffb.OP_FORWARD | ffb.OP_BACKWARD_DX | ffb.OP_GRAD_COEFF
    timeouts0 = ffb.framefb_wait_timeouts()
    batch = AdapterBatch(w, dev, ops=ops, indices=None if args.mats is None else range(args.mats))
    ws = batch.workspace(ops)
    stream = torch.cuda.current_stream()
    alg = algorithmic_bytes(batch)
    kernels = ffb.framefb_kernel_names(batch.mats, ops, batch.dtype_code)

    for _ in range(args.warmup):
        batch.run(ops, ws, stream)
    torch.cuda.synchronize()

    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t_start = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_start.record(stream)
        for a, b in evs:
            a.record(stream)
            batch.run(ops, ws, stream)
            b.record(stream)
        t_end.record(stream)
        torch.cuda.synchronize()
    barrier()
    total_ms = t_start.elapsed_time(t_end)
    kern_ms = [a.elapsed_time(b) for a, b in evs]
    ms_step = max_over_ranks(total_ms, world, dev) / args.steps
    value = w.N * world / (ms_step / 1e3)
    kernel_ms = statistics.mean(kern_ms)
    peak, peak_kind = peaks()
    achieved = alg / (kernel_ms / 1e3) / 1e9  # = bytes per launch / time per launch (equal launches)
    chunk = 64 if kernel_choice() in ("tc", "tc2") else 256
    launches = (len(batch.bufs) + chunk - 1) // chunk  # tile-kernel launches per step (each with a dC reduction)

    e2e = None
    if not args.no_e2e:
        e2e = e2e_timing(batch, ops, ws, stream, max(2, min(args.steps, 4)), world, dev, barrier)

    # the optimiser step on the coefficients of all matrices (one framefb_adamw
    # call over the contiguous [matrices x nnz] values), timed on its own after
    # the headline step: 16 bytes read and 12 written per coefficient
    opt = None
    if not args.no_optimizer:
        mo, vo = torch.zeros_like(batch.C), torch.zeros_like(batch.C)
        for t in range(1, 4):
            ffb.framefb_adamw(batch.C, batch.dC, mo, vo, t, 1e-3, stream=stream)
        o0 = torch.cuda.Event(enable_timing=True)
        o1 = torch.cuda.Event(enable_timing=True)
        reps = 200
        o0.record(stream)
        for t in range(4, 4 + reps):
            ffb.framefb_adamw(batch.C, batch.dC, mo, vo, t, 1e-3, stream=stream)
        o1.record(stream)
        torch.cuda.synchronize()
        us = o0.elapsed_time(o1) * 1e3 / reps
        nb = 28 * batch.C.numel()
        opt = {"kernel": "adamw_kernel", "us_per_call": us, "coefficients": batch.C.numel(), "bytes_per_call": nb,
               "achieved_gbs": nb / (us * 1e-6) / 1e9, "note": "arrays L2-resident between calls; launch-bound"}
        del mo, vo

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        k = min(args.cpu_mats, len(w.mats))
        tcpu, tsetup = cpu_oracle_sample(w, args.cpu_tokens, tuple(range(k)))
        cpu_tok = args.cpu_tokens / (tcpu / k * len(w.mats))
        cpu = {"value": cpu_tok, "unit": "tokens/s", "cores": cpu_threads(), "kind": "oracle",
               "sample": f"dense fp64 oracle on {k} of {len(w.mats)} matrices ({w.mats[0].m}x{w.mats[0].n}) over "
                         f"{args.cpu_tokens} tokens each ({tcpu:.1f} s), scaled to {len(w.mats)} matrices; frame and "
                         f"support setup ({tsetup:.1f} s) excluded", **host_info()}

    headline = (kernel_ms, alg, kernels)
    del batch, ws
    torch.cuda.empty_cache()

    serving = serving_timing(dev, stream) if args.serving else None

    per_config = None
    if rank == 0 and not args.no_per_config and args.mats is None and args.tokens is None:
        flush = L2Flush(dev)
        per_config = {}
        with_cpu = world == 1 and not args.no_cpu
        for name in [c for c in args.configs.split(",") if c]:
            per_config[name] = time_config(name, dev, stream, 5, 3, flush, with_cpu,
                                           headline if name == w.name else None)
        per_config["vit_b16_merge.merge"] = time_merge(dev, stream, 20, 3, flush)
        if "vit_b16_merge" in args.configs.split(","):
            per_config["vit_b16_merge.serving"] = serving if serving is not None else serving_timing(dev, stream)
        del flush
        torch.cuda.empty_cache()

    timeouts = ffb.framefb_wait_timeouts() - timeouts0

    if rank == 0:
        cfg = config_of(w, len(w.mats) if args.mats is None else args.mats, world)
        out = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
               "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
               "vs_baseline": None, "dtype": w.dtype, "data": "synthetic", "config": cfg,
               "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                            "frac": achieved / peak,
                            "traffic": (measured_traffic()
                                        if args.mats is None and args.workload is None and args.tokens is None else None),
                            "peak_kind": peak_kind,
                            "kernel": ",".join(kernels) + " + dc_reduce_kernel",
                            "kernel_ms": kernel_ms,
                            "algorithmic_bytes": alg, "algorithmic_bytes_per_launch": alg / launches,
                            "launches_per_step": launches, "frac_of_8tbs": achieved / NOMINAL_GBS},
               "cpu_baseline": cpu, "e2e": e2e, "optimizer": opt, "serving": serving, "per_config": per_config,
               "gpu_launches": 2 * launches * args.steps, "wait_timeouts": timeouts,
               "clocks": clk.summary()}
        print(json.dumps(out), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()

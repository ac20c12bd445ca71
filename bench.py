#!/usr/bin/env python
"""Benchmark of the W4A16 linear hot path on GB300.

Default step: one pass of the 175B-class int4 linear stack -- 96 layers x
{QKV 12288->36864, O 12288->12288, up 12288->49152, down 49152->12288},
g = 128, all ~88 GB of packed weights resident in HBM -- over a batch of 64
protein-ligand pairs x 1024 tokens (M = 65536).  `value` is scored pairs/s.

Other workloads (--config qkv | mlp_up | mlp_down | mlp_swiglu | gemv | tiny) print the
same JSON line for one linear (TFLOP/s, or GB/s for the small-M kernel).

--impl reference times the CPU oracle (the only reference there is) on a
bounded sample of the same workload on the host cores.

Multi-GPU (torchrun): the stack is replicated per GPU and the pairs are
data-parallel (no collective on the data path); value = pairs of all ranks
/ max-over-ranks time, scaling "weak".
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "W4A16 GEMM TFLOP/s & % of roofline; scored pairs/s on 175B-class linear stack"

# ncu DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum per launch) of
# the timed kernel, from the captures summarised in profiles/, keyed by the
# workload and by a hash of the kernel's sources at capture time: once the
# kernel changes the hash no longer matches and traffic is reported as null.
NCU_TRAFFIC = {
    # mean of one launch per stack shape at M = 16384 (384-token tiles, as in
    # the benched stack), scaled by 4 to M = 65536
    # (profiles/gemm_pair_wide_stack_traffic_m16384.md)
    ("stack", "ts", "cc26b2d7ce6a2d19"): 7.1208e9 * 4,
    # QKV prefill 4096x12288x36864 (384-token CTA pairs), one launch
    # (profiles/gemm_pair_wide_qkv_prefill_4096x12288x36864.md)
    ("qkv", "ts", "cc26b2d7ce6a2d19"): 1.4663e9 + 0.2894e9,
    # MLP up / down at 8192 tokens (384-token CTA pairs), one launch each
    # (DRAM counters only; profiles/gemm_pair_mlp_traffic_8192.md)
    ("mlp_up", "ts", "cc26b2d7ce6a2d19"): 3.9122e9 + 0.8025e9,
    ("mlp_down", "ts", "cc26b2d7ce6a2d19"): 4.7823e9 + 0.1976e9,
    # small-M readout, M = 8 (warp-level kernel), 12288x49152, one launch
    ("gemv", "gemv", "270f49f687deb1b3"): 0.31859e9 + 0.00380e9,
    # the same at M = 16 (16 token columns), one launch (DRAM counters only)
    ("gemv16", "gemv", "270f49f687deb1b3"): 0.31808e9 + 0.00319e9,
    # small-M readout, M = 32 (tensor-core kernel), 12288x49152, one launch
    ("gemv32", "gemvtc", "b81ddd27f1e19156"): 0.32655e9 + 0.00362e9,
    # attention prefill per 8 pairs of 1024 tokens x 96 heads (full capture of
    # one 8-pair launch); scaled by pairs / 8 for the benched launch
    ("attention", "attn", "f94e5ad5312cd435"): 0.8716e9 + 0.1923e9,
}

KERNEL_FILES = {"ts": ("ts_gemm.cu", "dequant.cuh", "ptx.cuh"),
                "gemv": ("gemv_rows.cu", "dequant.cuh", "ptx.cuh"),
                "gemvtc": ("gemv_tc.cu", "dequant.cuh", "ptx.cuh"),
                "attn": ("attention.cu",)}


def kernel_source_hash(kind: str = "ts") -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_30877_gb300", "csrc")
    for name in KERNEL_FILES[kind]:
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def ncu_traffic(config: str, m: int, pairs: int = 8):
    if config == "topk":
        return None  # no capture of the readout kernels is summarised
    if config == "attention":
        t = NCU_TRAFFIC.get((config, "attn", kernel_source_hash("attn")))
        return None if t is None else t * pairs / 8  # qkv and out grow with the pairs
    if config == "gemv":
        if 17 <= m <= 32:  # the tensor-core kernel; the capture is of M = 32
            return NCU_TRAFFIC.get(("gemv32", "gemvtc", kernel_source_hash("gemvtc")))
        if m > 8:  # the M = 9..16 instantiation, captured at M = 16
            return NCU_TRAFFIC.get(("gemv16", "gemv", kernel_source_hash("gemv")))
        kind = "gemv"
    else:
        kind = "ts"
    return NCU_TRAFFIC.get((config, kind, kernel_source_hash(kind)))


# The GB300's nominal dense bf16 tensor rate and HBM3e bandwidth: each
# roofline also carries its fraction of these (frac_nominal).
NOMINAL_BF16_TFLOPS = 2250.0
NOMINAL_HBM_GBS = 8000.0


def load_peaks() -> dict:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d["bf16_tflops_sustained"], "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


# ----------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        import tempfile
        fd, self.path = tempfile.mkstemp(prefix="clk_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self) -> dict:
        rows = []
        if self.path and os.path.exists(self.path):
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
            os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        def num(s):
            try:
                return float(s)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        smax = max(num(r[2]) or 0 for r in rows)
        power = [num(r[3]) for r in rows if num(r[3]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        loaded = [s for s in sm if s >= 0.5 * smax] or sm
        return {"sm_mhz": statistics.median(loaded) if loaded else None, "sm_max_mhz": smax,
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max(power) if power else None}


# ----------------------------------------------------------------- distributed

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def init_dist(world, local, backend="nccl"):
    """One process per GPU (nccl); gloo runs the same host logic on CPU."""
    import torch
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        if backend == "nccl":
            torch.cuda.set_device(local)
            dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        else:
            dist.init_process_group(backend)
    return dist if world > 1 else None


def _cuda_ok():
    import torch
    return torch.cuda.is_available()


def barrier(dist):
    import torch
    if dist is not None:
        dist.barrier()
    if _cuda_ok():
        torch.cuda.synchronize()


def max_over_ranks(dist, v: float) -> float:
    """The slowest rank's time: the job is done when every replica is."""
    import torch
    if dist is None:
        return v
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([v], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_value(world: int, units_per_step: float, step_s: float) -> float:
    """Whole-job throughput of N replicas (weak scaling): every rank runs the
    same per-GPU work, so units of all ranks over the slowest rank's time."""
    return world * units_per_step / step_s


# ----------------------------------------------------------------- workloads

def linear_flops(M, N, K):
    return 2.0 * M * N * K


def linear_bytes(M, N, K, g, n_out=None):
    """Algorithmic bytes of one linear: packed weights + scales + x once + out once."""
    n_out = N if n_out is None else n_out
    return N * K / 2 + 2.0 * N * (K // g) + 2.0 * M * K + 2.0 * M * n_out


def make_weights(N, K, g, seed):
    from paper_2608_30877_gb300 import synthetic as S
    from paper_2608_30877_gb300 import w4a16 as W
    w = S.make_w_master(N, K, seed, "cuda")
    packed, scales = W.quantize(w, g)
    del w
    return packed, scales


def _which(xs, t):
    for i, x in enumerate(xs):
        if x is t:
            return i
    raise ValueError("not an input buffer of the stack")


class StackWorkload:
    def __init__(self, pairs, tokens, layers, g=128, graph=False):
        import torch
        from paper_2608_30877_gb300 import synthetic as S
        from paper_2608_30877_gb300 import w4a16 as W
        self.M = pairs * tokens
        self.pairs = pairs
        self.layers = layers
        self.g = g
        self.flops = 0.0
        self.bytes = 0.0
        # one resident activation and output buffer per linear shape
        self.x = [S.make_x(self.M, K, 2000 + j, "cuda") for j, (_, K, _) in enumerate(S.LAYER_LINEARS)]
        self.out = [torch.empty((self.M, N), dtype=torch.bfloat16, device="cuda")
                    for (_, _, N) in S.LAYER_LINEARS]
        entries = []
        self.w = []
        for l in range(layers):
            for j, (_, K, N) in enumerate(S.LAYER_LINEARS):
                packed, scales = make_weights(N, K, g, 1000 + 4 * l + j)
                self.w.append((packed, scales))
                entries.append((self.x[j], packed, scales, self.out[j]))
                self.flops += linear_flops(self.M, N, K)
                self.bytes += linear_bytes(self.M, N, K, g)
        torch.cuda.synchronize()
        self.entries = entries
        self.arr = W.make_layer_array(entries)
        self.launches_per_step = len(entries)
        # one CUDA graph of the whole pass, replayed per step (w4a16_stack_graph_*)
        self.graph = W.StackGraph(entries, self.M, g) if graph else None

    def step(self, stream=None):
        from paper_2608_30877_gb300 import w4a16 as W
        if self.graph is not None:
            self.graph.launch(stream)
        else:
            W.linear_stack_array(self.arr, self.M, self.g, stream)

    def second_input_set(self):
        """A second set of input buffers and its layer array, so that the
        end-to-end loop can copy the next step's inputs during this step."""
        import torch
        from paper_2608_30877_gb300 import w4a16 as W
        x2 = [torch.empty_like(x) for x in self.x]
        entries = [(x2[_which(self.x, e[0])], e[1], e[2], e[3]) for e in self.entries]
        return x2, W.make_layer_array(entries)

    def per_linear(self, reps=3):
        """Event-timed TFLOP/s of each linear shape (layer 0), outside the timed region."""
        import torch
        from paper_2608_30877_gb300 import synthetic as S
        from paper_2608_30877_gb300 import w4a16 as W
        res = {}
        for j, (name, K, N) in enumerate(S.LAYER_LINEARS):
            x, packed, scales, out = self.entries[j]
            W.linear(x, packed, scales, self.g, out=out)
            ts = []
            for _ in range(reps):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record()
                W.linear(x, packed, scales, self.g, out=out)
                b.record()
                b.synchronize()
                ts.append(a.elapsed_time(b) / 1e3)
            t = statistics.median(ts)
            res[name] = {"ms": t * 1e3, "tflops": linear_flops(self.M, N, K) / t / 1e12}
        return res


class LinearWorkload:
    """One linear shape; for the small-M kernel the weights rotate over copies
    so that no launch finds its weights in L2."""

    def __init__(self, name, M, N, K, g, seed, copies=1, act=0):
        import torch
        from paper_2608_30877_gb300 import synthetic as S
        self.name, self.M, self.N, self.K, self.g, self.act = name, M, N, K, g, act
        self.x = S.make_x(M, K, seed, "cuda")
        n_out = N // 2 if act == 1 else N
        self.out = torch.empty((M, n_out), dtype=torch.bfloat16, device="cuda")
        self.w = [make_weights(N, K, g, seed + 10 * c) for c in range(copies)]
        self.flops = linear_flops(M, N, K)
        self.bytes = linear_bytes(M, N, K, g, n_out)
        self.launches_per_step = 1
        self.i = 0

    def step(self, stream=None):
        from paper_2608_30877_gb300 import w4a16 as W
        packed, scales = self.w[self.i % len(self.w)]
        self.i += 1
        if self.act:
            W.linear_fused(self.x, packed, scales, self.g, act=self.act, out=self.out,
                           stream=stream)
        else:
            W.linear(self.x, packed, scales, self.g, out=self.out, stream=stream)


class AttentionWorkload:
    """Attention prefill of one layer over the packed batch: `pairs` sequences
    of `tokens` tokens, 96 heads of 128, causal, 32K window; qkv resident."""

    def __init__(self, pairs, tokens, heads, window, seed):
        import torch
        from paper_2608_30877_gb300 import synthetic as S
        self.name = f"attention_{pairs}x{tokens}_h{heads}"
        M = pairs * tokens
        self.H, self.window = heads, window
        self.x = S.make_x(M, 3 * heads * 128, seed, "cuda")
        self.seq_start = torch.arange(0, M + 1, tokens, dtype=torch.int32, device="cuda")
        self.out = torch.empty((M, heads * 128), dtype=torch.bfloat16, device="cuda")
        keys = pairs * sum(min(i + 1, window) for i in range(tokens))  # allowed (i, j) pairs
        self.flops = 4.0 * 128 * heads * keys          # QK^T and PV, 2 flops per MAC
        self.bytes = 2.0 * M * 3 * heads * 128 + 2.0 * M * heads * 128
        self.launches_per_step = 1

    def step(self, stream=None):
        from paper_2608_30877_gb300 import w4a16 as W
        W.attention_prefill(self.x, self.seq_start, self.H, self.window, out=self.out,
                            stream=stream)


class TopkWorkload:
    """Result sorting of the screening set: the k best (smallest) of n
    predicted affinities, fp32 scores resident on the device."""

    def __init__(self, n, k, seed):
        import torch
        g = torch.Generator(device="cuda")
        g.manual_seed(seed)
        self.name, self.n, self.k = f"topk_n{n}_k{k}", n, k
        self.x = torch.randn(n, generator=g, device="cuda") * 2.0 - 8.0   # kcal/mol-like
        self.out = torch.empty(k, dtype=torch.float32, device="cuda")
        self.flops = 0.0
        self.bytes = 4.0 * n + 8.0 * k       # scores read once, (index, score) written once
        self.launches_per_step = 1

    def step(self, stream=None):
        from paper_2608_30877_gb300 import w4a16 as W
        _, self.out = W.topk_smallest(self.x, self.k, stream=stream)


# ----------------------------------------------------------------- CPU oracle

def oracle_sample(K: int, N_rows: int, target_s: float, rows_max: int = 2048):
    """Times the oracle on `r` token rows x N_rows weight rows of one K-deep
    linear with seeded inputs; grows r until the sample takes ~target_s.
    Returns (MAC/s, description, threads)."""
    import numpy as np
    from oracle import oracle as O
    from paper_2608_30877_gb300 import synthetic as S
    w = S.make_w_master(N_rows, K, 1000, "cpu").numpy()
    packed, scales = O.quantize(w, 128)
    x = S.bf16_bits(S.make_x(rows_max, K, 2000, "cpu"))
    threads = len(os.sched_getaffinity(0))
    r, spent, macs = 1, 0.0, 0
    while True:
        t0 = time.perf_counter()
        O.linear_rows(x[:r], packed, scales, N_rows, K, 128, nthreads=threads)
        dt = time.perf_counter() - t0
        spent += dt
        macs_r = r * N_rows * K
        if dt >= target_s / 3 or r >= rows_max or spent >= 2 * target_s:
            desc = (f"oracle fp64 linear, {r} token rows x {N_rows} weight rows x K={K} "
                    f"({macs_r / 1e9:.2f} GMAC) in {dt:.2f} s on {threads} threads")
            return macs_r / dt, desc, threads
        r = min(rows_max, max(r + 1, int(r * (target_s / 2) / max(dt, 1e-3))))


def oracle_attention_sample(target_s: float = 10.0):
    """Times the oracle's fp64 attention on query rows of one 1024-token
    sequence with 96 heads of 128 (rows taken from the end, the longest),
    growing the row count toward target_s; returns (TFLOP/s, description)."""
    import numpy as np
    from oracle import oracle as O
    from paper_2608_30877_gb300 import synthetic as S
    H, L = 96, 1024
    bits = S.bf16_bits(S.make_x(L, 3 * H * 128, 9, "cpu"))
    st = np.array([0, L], dtype=np.int64)
    r = 1
    while True:
        rows = np.arange(L - r, L, dtype=np.int64)
        t0 = time.perf_counter()
        O.attention_rows(bits, H, 128, st, 32768, rows=rows)
        dt = time.perf_counter() - t0
        if dt >= target_s / 3 or r >= 256:
            flops = 4.0 * 128 * H * float(np.sum(rows + 1))
            return flops / dt / 1e12, (f"oracle fp64 attention, {r} query rows of a 1024-token "
                                       f"sequence x 96 heads in {dt:.2f} s on 1 thread")
        r = min(256, max(r + 1, int(r * (target_s / 2) / max(dt, 1e-3))))


def oracle_topk_sample(n: int, k: int):
    """Times the oracle's top-k (plain repeated selection, one thread) on the
    same n seeded scores with k reduced to fit ~10 s; returns (GB/s of the
    algorithmic bytes 4 n + 8 k scaled to the full k, description)."""
    import numpy as np
    from oracle import oracle as O
    s = (np.random.default_rng(5).normal(size=n) * 2.0 - 8.0).astype(np.float32)
    kk = max(1, min(k, 50))
    t0 = time.perf_counter()
    O.topk_smallest(s, kk)
    dt = time.perf_counter() - t0
    t_full = dt * k / kk                  # selection time grows linearly in k
    desc = (f"oracle top-k by repeated selection, n={n}, k={kk} in {dt:.2f} s on 1 thread, "
            f"scaled linearly to k={k}")
    return (4.0 * n + 8.0 * k) / t_full / 1e9, desc


def stack_macs_per_pair(tokens=1024, layers=96):
    from paper_2608_30877_gb300 import synthetic as S
    return tokens * layers * sum(N * K for (_, K, N) in S.LAYER_LINEARS)


# ----------------------------------------------------------------- main

def config_for(args):
    from paper_2608_30877_gb300 import synthetic as S
    c = args.config
    if c == "stack":
        return {"workload": "175B-class int4 linear stack, 96 layers x {qkv 12288->36864, "
                            "o 12288->12288, up 12288->49152, down 49152->12288}, "
                            f"M={args.pairs * args.tokens} ({args.pairs} pairs x {args.tokens} tokens), "
                            "g=128" + (", replayed as one CUDA graph" if args.graph else ""),
                "pairs": args.pairs, "tokens_per_pair": args.tokens, "layers": args.layers, "g": 128,
                "graph": bool(args.graph),
                "activations": "one resident seeded input per linear shape (4 buffers, seeds "
                               "2000..2003) read by all 96 layers, instead of a fresh input per "
                               "layer; each is larger than L2, so the reuse leaves the timed work "
                               "unchanged; the e2e leg copies those 4 buffers in per step",
                "l2": "inputs larger than L2 (88 GB packed weights, >=1.6 GB activations per "
                      "linear); no flush"}
    if c == "attention":
        return {"workload": f"attention prefill, {args.pairs} pairs x 1024 tokens, 96 heads x 128, "
                            "causal, window 32768",
                "pairs": args.pairs, "tokens_per_pair": 1024, "heads": 96, "head_dim": 128,
                "window": 32768, "l2": "qkv (4.8 GB at 64 pairs) larger than L2; no flush"}
    if c == "topk":
        return {"workload": f"top-k of predicted affinities, n={args.topk_n}, k={args.topk_k}",
                "n": args.topk_n, "k": args.topk_k,
                "l2": "scores (<1 MB) stay in L2: the step is latency-bound; no flush"}
    cases = {"qkv": S.QKV_PREFILL, "mlp_up": S.MLP_UP, "mlp_down": S.MLP_DOWN, "tiny": S.TINY,
             "mlp_swiglu": S.MLP_SWIGLU}
    if c == "gemv":
        lc = S.gemv_case(args.m)
    else:
        lc = cases[c]
    cfg = {"workload": lc.name, "M": lc.M, "N": lc.N, "K": lc.K, "g": lc.g,
           "l2": "weights rotate over 2 copies larger than L2" if c == "gemv"
           else "inputs larger than L2; no flush"}
    if c == "mlp_swiglu":
        cfg["epilogue"] = "SwiGLU over interleaved gate/up rows, output N/2 columns"
    return cfg


def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return 0
    from paper_2608_30877_gb300 import synthetic as S
    if args.config == "attention":
        vals, desc = [], ""
        for i in range(args.warmup + args.steps):
            tf, desc = oracle_attention_sample(args.ref_seconds)
            if i >= args.warmup:
                vals.append(tf)
        value = statistics.median(vals)
        step_flops = 4.0 * 128 * 96 * args.pairs * (1024 * 1025 / 2)
        line = {"metric": METRIC, "impl": "reference", "value": value, "unit": "TFLOP/s",
                "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": 1e3 * step_flops / (value * 1e12),
                "ms_per_step_kind": "extrapolated from the timed sample's rate",
                "higher_is_better": True,
                "scaling": "weak",
                "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": config_for(args),
                "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": 1, "kind": "oracle",
                                 "sample": desc},
                "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line), flush=True)
        return 0
    if args.config == "topk":
        vals, desc = [], ""
        for i in range(args.warmup + args.steps):
            gbs, desc = oracle_topk_sample(args.topk_n, args.topk_k)
            if i >= args.warmup:
                vals.append(gbs)
        value = statistics.median(vals)
        line = {"metric": METRIC, "impl": "reference", "value": value, "unit": "GB/s",
                "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": 1e3 * (4.0 * args.topk_n + 8.0 * args.topk_k) / value / 1e9,
                "ms_per_step_kind": "extrapolated from the timed sample's rate",
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "f32", "data": "synthetic", "config": config_for(args),
                "cpu_baseline": {"value": value, "unit": "GB/s", "cores": 1, "kind": "oracle",
                                 "sample": desc},
                "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line), flush=True)
        return 0
    if args.config == "stack":
        K, N_rows = S.D_MODEL, 2048
        unit = "pairs/s"
        per_unit = stack_macs_per_pair(args.tokens, args.layers)
    else:
        cfg = config_for(args)
        K, N_rows = cfg["K"], min(cfg["N"], 2048)
        unit = "TFLOP/s"
        per_unit = None
    vals = []
    desc, threads = "", 1
    for i in range(args.warmup + args.steps):
        mac_s, desc, threads = oracle_sample(K, N_rows, target_s=args.ref_seconds)
        if i >= args.warmup:
            vals.append(mac_s)
    mac_s = statistics.median(vals)
    value = mac_s / per_unit if per_unit else 2 * mac_s / 1e12
    step_ms = 1e3 * (per_unit / mac_s if per_unit else 0)
    line = {"metric": METRIC, "impl": "reference", "value": value, "unit": unit, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_ms,
            "ms_per_step_kind": "extrapolated: the workload's MACs over the oracle's MAC rate on "
                                "the timed sample (one step of the whole workload is never run)",
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": config_for(args),
            "cpu_baseline": {"value": value, "unit": unit, "cores": threads, "kind": "oracle",
                             "sample": desc},
            "e2e": {"value": value, "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="stack",
                    choices=["stack", "qkv", "mlp_up", "mlp_down", "mlp_swiglu", "gemv", "tiny",
                             "topk", "attention"])
    ap.add_argument("--topk-n", type=int, default=200000, help="scores for --config topk")
    ap.add_argument("--topk-k", type=int, default=1000, help="k for --config topk")
    ap.add_argument("--m", type=int, default=32, help="tokens for --config gemv")
    ap.add_argument("--pairs", type=int, default=64)
    ap.add_argument("--tokens", type=int, default=1024, help="tokens per pair for the stack")
    ap.add_argument("--graph", action="store_true",
                    help="replay the stack as one captured CUDA graph")
    ap.add_argument("--layers", type=int, default=96)
    ap.add_argument("--ref-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the QKV / MLP / small-M workloads timed after the stack")
    args = ap.parse_args()
    if args.warmup < 3:
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)
    if args.impl == "reference":
        return run_reference(args)

    import torch
    world, rank, local = dist_env()
    torch.cuda.set_device(local)
    dist = init_dist(world, local)
    from paper_2608_30877_gb300 import w4a16 as W
    W.lib()
    peaks = load_peaks()

    setup_t0 = time.perf_counter()
    if args.config == "stack":
        wl = StackWorkload(args.pairs, args.tokens, args.layers, graph=args.graph)
        unit = "pairs/s"
        units_per_step = wl.pairs
    elif args.config == "topk":
        wl = TopkWorkload(args.topk_n, args.topk_k, 5)
        unit = "GB/s"
        units_per_step = None
    elif args.config == "attention":
        wl = AttentionWorkload(args.pairs, 1024, 96, 32768, 9)
        unit = "TFLOP/s"
        units_per_step = None
    else:
        from paper_2608_30877_gb300 import synthetic as S
        cfg = config_for(args)
        copies = 2 if args.config == "gemv" else 1
        wl = LinearWorkload(cfg["workload"], cfg["M"], cfg["N"], cfg["K"], cfg["g"], 3, copies,
                            act=1 if args.config == "mlp_swiglu" else 0)
        unit = "GB/s" if args.config == "gemv" else "TFLOP/s"
        units_per_step = None
    setup_s = time.perf_counter() - setup_t0

    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        wl.step()
    barrier(dist)

    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    gpu_index = torch.cuda.current_device() if "CUDA_VISIBLE_DEVICES" not in os.environ else local
    with ClockSampler(gpu_index) as clk:
        barrier(dist)
        start.record(stream)
        for _ in range(args.steps):
            wl.step()
        end.record(stream)
        end.synchronize()
        barrier(dist)
    elapsed = start.elapsed_time(end) / 1e3
    elapsed = max_over_ranks(dist, elapsed)
    step_s = elapsed / args.steps
    if W.get_device_error() != W.OK:
        raise RuntimeError("device status word set during the timed region")

    if args.config == "stack":
        value = replica_value(world, units_per_step, step_s)
    elif args.config in ("gemv", "topk"):
        value = world * wl.bytes / step_s / 1e9
    else:
        value = world * wl.flops / step_s / 1e12

    # roofline of the fused kernel: every launch in the step is that kernel
    per_launch_s = step_s / wl.launches_per_step
    if args.config in ("gemv", "topk"):
        achieved = wl.bytes / step_s / 1e9
        peak = peaks["hbm_gbs"]
        roof = {"bound": "hbm", "unit": "GB/s"}
    else:
        achieved = wl.flops / step_s / 1e12
        peak = peaks["bf16_tflops_sustained"] if args.config == "stack" else peaks["bf16_tflops"]
        roof = {"bound": "tensor", "unit": "TFLOP/s"}
    traffic = ncu_traffic(args.config, args.m, args.pairs)
    nominal = NOMINAL_HBM_GBS if roof["bound"] == "hbm" else NOMINAL_BF16_TFLOPS
    roof.update({"achieved": achieved, "peak": peak, "frac": achieved / peak,
                 "frac_nominal": achieved / nominal,
                 "traffic": traffic, "peak_source": peaks["source"] + (
                     " bf16_tflops_sustained" if args.config == "stack" else
                     (" hbm_gbs" if args.config in ("gemv", "topk") else " bf16_tflops")),
                 "per_launch_ms": per_launch_s * 1e3,
                 "algorithmic_bytes_per_step": wl.bytes, "flops_per_step": wl.flops})

    line = {"metric": METRIC, "value": value, "unit": unit, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": step_s * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": config_for(args), "clocks": clk.summary(), "roofline": roof,
            "gpu_launches": wl.launches_per_step * args.steps, "setup_s": setup_s}
    if args.config == "stack":
        line["tflops"] = wl.flops / step_s / 1e12
        if rank == 0:
            line["per_linear"] = wl.per_linear()

    # end to end through the public API with host buffers
    if not args.no_e2e:
        line["e2e"] = e2e(wl, args, dist, world, unit, units_per_step)

    # the other named workloads, at N = 1 after the stack (its buffers freed)
    if args.config == "stack" and world == 1 and not args.no_configs:
        del wl
        torch.cuda.empty_cache()
        line["configs"] = configs_sweep(peaks, gpu_index)

    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from paper_2608_30877_gb300 import synthetic as S
        if args.config == "topk":
            gbs, desc = oracle_topk_sample(args.topk_n, args.topk_k)
            line["cpu_baseline"] = {"value": gbs, "unit": "GB/s", "cores": 1, "kind": "oracle",
                                    "sample": desc}
        elif args.config == "attention":
            tf, desc = oracle_attention_sample()
            line["cpu_baseline"] = {"value": tf, "unit": "TFLOP/s", "cores": 1, "kind": "oracle",
                                    "sample": desc}
        elif args.config == "stack":
            mac_s, desc, threads = oracle_sample(S.D_MODEL, 2048, 15.0)
            cb = mac_s / stack_macs_per_pair(args.tokens, args.layers)
            line["cpu_baseline"] = {"value": cb, "unit": "pairs/s", "cores": threads,
                                    "kind": "oracle", "sample": desc}
        else:
            cfg = config_for(args)
            mac_s, desc, threads = oracle_sample(cfg["K"], min(cfg["N"], 2048), 15.0)
            if args.config == "gemv":
                cb = (wl.bytes / (cfg["M"] * cfg["N"] * cfg["K"] / mac_s)) / 1e9
                cu = "GB/s"
            else:
                cb, cu = 2 * mac_s / 1e12, "TFLOP/s"
            line["cpu_baseline"] = {"value": cb, "unit": cu, "cores": threads,
                                    "kind": "oracle", "sample": desc}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def _timed_reps(wl, gpu, warmup, seconds):
    """Times wl.step() alone (CUDA events on the launching stream, clocks
    sampled meanwhile): warm-up launches, the last two timed to size the timed
    region at about `seconds` (so that the clock sampler sees it), then 10
    back-to-back repetitions, each bracketed by its own events.  Returns the
    mean time per launch over all of them, the launch count, and the
    per-launch spread over the repetitions and the clock summary as dicts."""
    import torch
    stream = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(gpu) as clk:
        for _ in range(warmup - 2):
            wl.step()
        a.record(stream)
        for _ in range(2):
            wl.step()
        b.record(stream)
        b.synchronize()
        reps = 10
        per_rep = max(1, int(seconds / (a.elapsed_time(b) / 2e3)) // reps)
        steps = reps * per_rep
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(reps + 1)]
        ev[0].record(stream)
        for r in range(reps):
            for _ in range(per_rep):
                wl.step()
            ev[r + 1].record(stream)
        ev[-1].synchronize()
    rep_us = sorted(ev[r].elapsed_time(ev[r + 1]) * 1e3 / per_rep for r in range(reps))
    t = ev[0].elapsed_time(ev[-1]) / 1e3 / steps
    spread = {"reps": reps, "launches_per_rep": per_rep,
              "median": (rep_us[reps // 2 - 1] + rep_us[reps // 2]) / 2,
              "min": rep_us[0], "max": rep_us[-1]}
    return t, steps, spread, clk.summary()


def _config_line(workload, wl, t, steps, spread, clocks, peaks, hbm, traffic, l2):
    if hbm:
        ach, peak, unit = wl.bytes / t / 1e9, peaks["hbm_gbs"], "GB/s"
    else:
        ach, peak, unit = wl.flops / t / 1e12, peaks["bf16_tflops"], "TFLOP/s"
    return {"workload": workload, "value": ach, "unit": unit, "us_per_launch": t * 1e6,
            "launches": steps, "us_per_launch_reps": spread, "clocks": clocks,
            "roofline": {"bound": "hbm" if hbm else "tensor", "achieved": ach, "peak": peak,
                         "unit": unit, "frac": ach / peak,
                         "frac_nominal": ach / (NOMINAL_HBM_GBS if hbm else NOMINAL_BF16_TFLOPS),
                         "traffic": traffic,
                         "peak_source": peaks["source"] + (" hbm_gbs" if hbm else " bf16_tflops"),
                         "algorithmic_bytes": wl.bytes, "flops": wl.flops},
            "l2": l2}


def time_linear_config(name, lc, peaks, gpu, warmup, copies=1, seconds=1.2):
    """One linear workload timed alone, with its own roofline: TFLOP/s
    against the measured bf16 burst peak for the GEMMs, GB/s against the
    measured copy bandwidth for the small-M readout."""
    import torch
    from paper_2608_30877_gb300 import w4a16 as W
    wl = LinearWorkload(lc.name, lc.M, lc.N, lc.K, lc.g, lc.w_seed, copies)
    t, steps, spread, clocks = _timed_reps(wl, gpu, warmup, seconds)
    if W.get_device_error() != W.OK:
        raise RuntimeError(f"device status word set during {name}")
    hbm = lc.M <= 32
    traffic = (ncu_traffic("gemv", lc.M) if hbm else
               ncu_traffic({"qkv_prefill": "qkv"}.get(name, name), lc.M))
    res = _config_line(lc.name, wl, t, steps, spread, clocks, peaks, hbm, traffic,
                       "weights rotate over 2 copies larger than L2" if copies > 1
                       else "inputs larger than L2; no flush")
    del wl
    torch.cuda.empty_cache()
    return res


def time_attention_config(peaks, gpu, pairs=64, seconds=1.2):
    """One attention prefill layer over the packed batch (64 pairs x 1024
    tokens, 96 heads of 128, causal, 32K window) timed alone: TFLOP/s against
    the measured bf16 burst peak."""
    import torch
    from paper_2608_30877_gb300 import w4a16 as W
    wl = AttentionWorkload(pairs, 1024, 96, 32768, 9)
    t, steps, spread, clocks = _timed_reps(wl, gpu, 4, seconds)
    if W.get_device_error() != W.OK:
        raise RuntimeError("device status word set during attention")
    res = _config_line(f"attention_prefill_{pairs}x1024_h96_w32768", wl, t, steps, spread,
                       clocks, peaks, False, ncu_traffic("attention", 0, pairs),
                       "qkv (4.8 GB at 64 pairs) larger than L2; no flush")
    del wl
    torch.cuda.empty_cache()
    return res


def configs_sweep(peaks, gpu):
    """The other named workloads, each timed alone after the stack: the
    QKV prefill, the MLP up and down projections (tensor-bound), the small-M
    readout at M = 1, 8, 16, 32 (HBM-bound) and one attention prefill layer
    (tensor-bound)."""
    from paper_2608_30877_gb300 import synthetic as S
    out = {}
    for key, lc in (("qkv_prefill", S.QKV_PREFILL), ("mlp_up", S.MLP_UP),
                    ("mlp_down", S.MLP_DOWN)):
        out[key] = time_linear_config(key, lc, peaks, gpu, warmup=4)
    for m in S.GEMV_MS:
        out[f"gemv_m{m}"] = time_linear_config(f"gemv_m{m}", S.gemv_case(m), peaks, gpu,
                                               warmup=6, copies=2)
    out["attention_prefill"] = time_attention_config(peaks, gpu)
    return out


def e2e_stack(wl, args, dist, world, unit, units_per_step):
    """e2e for the stack with double-buffered inputs: each step's inputs are
    copied from pinned host memory into one of two buffer sets on a copy
    stream while the previous step computes on the other set; every copy and
    every result read-back lies inside the timed region."""
    import torch
    from paper_2608_30877_gb300 import w4a16 as W
    srcs = [torch.empty_like(x, device="cpu").pin_memory() for x in wl.x]
    for s_, x in zip(srcs, wl.x):
        s_.copy_(x)
    x2, arr2 = wl.second_input_set()
    sets, arrs = [wl.x, x2], [wl.arr, arr2]
    result = wl.out[-1]
    host_out = torch.empty_like(result, device="cpu").pin_memory()
    h2d = sum(s_.numel() * s_.element_size() for s_ in srcs)
    d2h = host_out.numel() * host_out.element_size()
    comp, copy = torch.cuda.current_stream(), torch.cuda.Stream()
    copied = [torch.cuda.Event(), torch.cuda.Event()]
    done = [torch.cuda.Event(), torch.cuda.Event()]

    def copy_in(k):
        with torch.cuda.stream(copy):
            if k >= 2:
                copy.wait_event(done[k % 2])     # step k-2 has read this set
            for s_, d in zip(srcs, sets[k % 2]):
                d.copy_(s_, non_blocking=True)
            copied[k % 2].record(copy)

    def run(k):
        comp.wait_event(copied[k % 2])
        W.linear_stack_array(arrs[k % 2], wl.M, wl.g, comp)
        done[k % 2].record(comp)
        host_out.copy_(result, non_blocking=True)

    def loop(n, start=None):
        if start is not None:
            copy.wait_event(start)
        copy_in(0)
        for k in range(n):
            if k + 1 < n:
                copy_in(k + 1)
            run(k)

    loop(1)
    torch.cuda.synchronize()
    barrier(dist)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    steps = max(1, min(args.steps, 3))
    a.record(comp)
    loop(steps, a)
    b.record(comp)
    b.synchronize()
    t = max_over_ranks(dist, a.elapsed_time(b) / 1e3) / steps
    return {"value": replica_value(world, units_per_step, t), "unit": unit,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": steps,
            "overlap": "next step's inputs copied during this step (two buffer sets)"}


def e2e(wl, args, dist, world, unit, units_per_step):
    """Same metric, host buffers: per step the step's inputs are copied from
    pinned host memory, the library runs, and the result is read back."""
    import torch
    if isinstance(wl, StackWorkload) and wl.graph is None:
        return e2e_stack(wl, args, dist, world, unit, units_per_step)
    if isinstance(wl, StackWorkload):
        srcs = [torch.empty_like(x, device="cpu").pin_memory() for x in wl.x]
        for s, x in zip(srcs, wl.x):
            s.copy_(x)
        result = wl.out[-1]
    else:
        srcs = [torch.empty_like(wl.x, device="cpu").pin_memory()]
        srcs[0].copy_(wl.x)
        result = wl.out
    dsts = wl.x if isinstance(wl, StackWorkload) else [wl.x]
    host_out = torch.empty_like(result, device="cpu").pin_memory()
    h2d = sum(s.numel() * s.element_size() for s in srcs)
    d2h = host_out.numel() * host_out.element_size()

    def one():
        for s, d in zip(srcs, dsts):
            d.copy_(s, non_blocking=True)
        wl.step()
        host_out.copy_(result, non_blocking=True)

    one()
    barrier(dist)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    steps = max(1, min(args.steps, 2)) if isinstance(wl, StackWorkload) else args.steps
    a.record()
    for _ in range(steps):
        one()
    b.record()
    b.synchronize()
    t = max_over_ranks(dist, a.elapsed_time(b) / 1e3) / steps
    if isinstance(wl, StackWorkload):
        v = world * units_per_step / t
    elif unit == "GB/s":
        v = world * wl.bytes / t / 1e9
    else:
        v = world * wl.flops / t / 1e12
    return {"value": v, "unit": unit, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "steps": steps}


if __name__ == "__main__":
    sys.exit(main())

"""Benchmark of one ReTrace round (verify + align/refine + gated fusion) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--config 5]

A step is one retrace_round over one batch of the serving workload (default:
B=256 sequences, K=16 drafts, V=151936, d=4096, bf16; synthetic seeded
inputs resident in HBM).  L2 is flushed (256 MB write) before every timed
step and each step is timed on its stream with CUDA events; `value` is
rounds/s over the K timed steps, max over ranks.  K more timed steps record
the library's phase events inside each round (verification | conditioning)
for the per-kernel durations of the rooflines; an event between two kernels
keeps the second from starting early, so those steps are slightly slower
(`ms_per_step_with_phase_events`) and do not enter `value`.  Under torchrun every rank
runs its own batch on its own GPU (sequences are independent, so the ranks
shard the batch dimension with no data-path collective: weak scaling).

Also reported on the same JSON line:
  roofline_verify        the verification kernel (HBM-bound): algorithmic bytes
                per launch / its CUDA-event duration, against the measured HBM
                copy peak;
  roofline_conditioning  the projection kernel (tensor-bound): algorithmic
                flops / its duration, against the measured bf16 peak;
  roofline      whichever of the two takes the larger share of the round;
  e2e           the same metric through the public API with host buffers: the
                step's inputs copied from pinned host memory and its outputs
                read back inside the timed region;
  cpu_baseline  the CPU oracle timed on a bounded sample of the workload
                (rank 0, N = 1 only);
  clocks        nvidia-smi samples taken during the timed region.
`--impl reference` times the CPU oracle itself on this workload (the paper
has no code to run) and prints the same line with "impl": "reference".
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

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2608_29748_gb300.workloads import CONFIGS, PROFILE_CONFIG, RoundConfig, make_round_inputs  # noqa: E402

METRIC = "verify+ReTrace rounds/sec at 1 GB300; logits HBM GB/s and % of roofline"
UNIT = "rounds/s"
KERNELS_PER_ROUND_FUSED = 1  # cond_kernel<FUSED>: the whole round
KERNELS_PER_ROUND = 2  # one-pass verify_kernel (+ row packing), cond_kernel (both projections + gate-bias GEMV)
L2_FLUSH_BYTES = 256 << 20
# DRAM traffic per round (ncu dram__bytes_read.sum + dram__bytes_write.sum,
# summed over the kernels of the phase) of the phase a roofline object names,
# measured once with ncu on that workload.  Each figure holds only for the
# kernel sources it was measured on: `sources` is kernel_sources_hash() at the
# time, and the line reports null traffic once the sources differ.
TRAFFIC = {
    ("verify", "qwen3-8b-B256-K16"): {"bytes": 311308288 + 2800384 + 184310272 + 138752 + 55403264 + 0
                                      + 47179520 + 4033792, "sources": "c403a58964d4ce6e"},
    ("conditioning", "qwen3-8b-B256-K16"): {"bytes": 509979136 + 37198080, "sources": "c403a58964d4ce6e"},
}


def kernel_sources_hash() -> str:
    """Hash of every CUDA source of the library (kernels and their headers)."""
    import hashlib

    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_29748_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h")):
            with open(os.path.join(csrc, name), "rb") as f:
                h.update(name.encode() + b"\0" + f.read())
    return h.hexdigest()[:16]


def measured_traffic(phase: str, workload_name: str, variant: str) -> int | None:
    """ncu DRAM bytes per round of `phase` on this workload, if measured on
    the current kernel sources (the default, corrected variant only)."""
    t = TRAFFIC.get((phase, workload_name))
    if variant != "corrected" or t is None or t["sources"] != kernel_sources_hash():
        return None
    return t["bytes"]


# ---------------------------------------------------------------------------
# distributed plumbing (host side; testable with gloo on CPU)
# ---------------------------------------------------------------------------


def dist_env() -> tuple[int, int, int]:
    """(rank, local_rank, world_size) from the torchrun environment."""
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


def shard_seed(base_seed: int, rank: int) -> int:
    """Each rank draws its own batch: independent sequences, no shared data."""
    return base_seed + 7919 * rank


def max_over_ranks(x: float, world: int, device=None) -> float:
    if world <= 1:
        return x
    import torch.distributed as dist

    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int) -> None:
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def aggregate_value(rounds_per_rank: int, world: int, seconds_max: float) -> float:
    """Whole-job rounds/s: rounds of all ranks over the slowest rank's time."""
    return rounds_per_rank * world / seconds_max


# ---------------------------------------------------------------------------
# measurement helpers
# ---------------------------------------------------------------------------


def load_peaks() -> dict:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": p["hbm_gbs"], "bf16_tflops": p["bf16_tflops"],
                "bf16_tflops_sustained": p["bf16_tflops_sustained"], "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 20 ms while running."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "20"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self) -> dict | None:
        if not self.path or not os.path.exists(self.path):
            return None
        rows = []
        for line in open(self.path):
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
        reasons = sorted({names[i] for _, _, flags in rows for i, f in enumerate(flags) if f.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


def cpu_threads() -> int:
    for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(var, "").isdigit():
            return int(os.environ[var])
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


def prepare_oracle_sample(cfg: RoundConfig, sample_B: int, seed: int, lowrank: bool = False,
                          sampled: bool = False) -> dict:
    """Host float64 inputs for `sample_B` sequences drawn like `cfg` (weights at full size)."""
    from oracle import bf16_bits_to_f64  # test infrastructure: CPU-baseline legs only
    from paper_2608_29748_gb300.workloads import as_bits_numpy

    sub = RoundConfig(cfg.name + f"-sample{sample_B}", sample_B, cfg.K, cfg.V, cfg.d, cfg.dtype, cfg.logits_std,
                      cfg.prefix, cfg.prefix_p, cfg.ties, cfg.seed_offset)
    x = make_round_inputs(sub, device="cpu", seed=seed)

    def f64(t):
        return bf16_bits_to_f64(as_bits_numpy(t)) if t.dtype == torch.bfloat16 else t.double().numpy()

    host = {k: f64(x[k]) for k in ("logits", "hD", "hT", "e", "Wc", "Wv", "Wg")}
    host.update(draft=x["draft"].numpy(), beta=x["beta"], dtype=cfg.dtype, B=sample_B)
    if lowrank:
        from paper_2608_29748_gb300.workloads import make_lowrank_weights

        host["lowrank"] = {k: f64(v) for k, v in make_lowrank_weights(cfg, device="cpu").items()}
    if sampled:
        from paper_2608_29748_gb300.workloads import make_sampled_inputs

        sm = make_sampled_inputs(sub, x["logits"], device="cpu", seed=seed + 1)
        host["sampled"] = {"draft_logits": f64(sm["draft_logits"]), "draft": sm["draft"].numpy(),
                           "uniforms": sm["uniforms"].double().numpy(), "T": sm["temperature"], "k": sm["top_k"],
                           "p": sm["top_p"]}
    return host


def time_oracle(host: dict, variant: str = "corrected") -> float:
    """Seconds the CPU oracle takes for one round over the prepared sample."""
    # test infrastructure: CPU-baseline legs only
    from oracle import retrace_round as oracle_round_fn, retrace_round_lowrank as oracle_lowrank_fn

    t0 = time.perf_counter()
    if "sampled" in host:
        import oracle

        sm = host["sampled"]
        out = oracle.verify_sampled(host["logits"], sm["draft_logits"], sm["draft"], sm["uniforms"], sm["T"], sm["k"],
                                    sm["p"])
        K = sm["draft"].shape[1]
        m, u = oracle.align(host["hD"], host["hT"], out["accept_len"])
        e_full = np.broadcast_to(host["e"], host["hD"].shape)
        oracle.condition(e_full, m, u, oracle.carried_rows(out["accept_len"], K), host["Wc"], host["Wv"], host["Wg"],
                         host["beta"], "corrected", host["dtype"] == "bf16")
    elif "lowrank" in host:
        w = host["lowrank"]
        oracle_lowrank_fn(host["logits"], host["draft"], host["hD"], host["hT"], host["e"], w["P"], w["Bc"],
                          w["Ac"], w["Wv_lr"], w["Wg_lr"], host["beta"], host["dtype"])
    else:
        oracle_round_fn(host["logits"], host["draft"], host["hD"], host["hT"], host["e"], host["Wc"], host["Wv"],
                        host["Wg"], host["beta"], host["dtype"], variant=variant)
    return time.perf_counter() - t0


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------


VARIANT_FLAGS = {"corrected": 0, "raw": 0x2, "overwrite": 0x4, "none": 0x8}  # include/retrace.h
ROUND_OVERLAP_FLAG = 0x1


def needed_logits_bytes(cfg: RoundConfig, accept: np.ndarray) -> int:
    """Logits the verification outputs depend on: rows 0..A_b of each
    sequence (the argmaxes of later rows change nothing)."""
    return int(np.sum(accept.astype(np.int64) + 1)) * cfg.V * cfg.elem_bytes


def read_logits_bytes(cfg: RoundConfig, accept: np.ndarray, windows: list[int]) -> int:
    """Logits a greedy verification schedule streams: window k's rows for the
    sequences whose draft tokens matched every row before it."""
    rows = 0
    for k in range(len(windows) - 1):
        rows += int(np.sum(accept >= windows[k])) * (windows[k + 1] - windows[k])
    return rows * cfg.V * cfg.elem_bytes


def verify_bytes(cfg: RoundConfig, n: np.ndarray, packs_rows: bool, variant: str = "corrected",
                 accept: np.ndarray | None = None) -> int:
    """Algorithmic bytes of the verification phase of a round: the logits rows
    the outputs depend on, tokens, and the row copies / packing."""
    es = cfg.elem_bytes
    B, K, V, d = cfg.B, cfg.K, cfg.V, cfg.d
    logits = needed_logits_bytes(cfg, accept) if accept is not None else B * (K + 1) * V * es
    tokens_in = B * K * 4
    tokens_out = B * (K + 1) * 4 + 3 * B * 4  # committed; accept_len, bonus, n
    R = int(np.sum(n))
    if variant in ("overwrite", "none"):  # verification writes every row of e~
        copies = B * K * d * es + (R * d * es if variant == "overwrite" else 0)  # + the m rows read
        return logits + tokens_in + tokens_out + copies
    copies = int(np.sum(K - n)) * d * es  # unconditioned rows of e~ written
    packing = (2 * R * 2 * d * es + R * 4) if packs_rows else 0  # [m; u] rows read + written, row map
    return logits + tokens_in + tokens_out + copies + packing


def conditioning_flops(cfg: RoundConfig, R: int, dense_e: bool, variant: str = "corrected") -> int:
    d = cfg.d
    if variant in ("overwrite", "none"):
        return 0
    f = 2 * R * (2 * d) * d if variant == "corrected" else 0  # c = W_c [m; u]
    f += 2 * R * d * (2 * d)  # [v; g_r] = [W_v; W_g,r] r
    f += 2 * R * d * d if dense_e else 2 * d * d  # W_g,e e (per row, or once for a broadcast e)
    return f


LOWRANK_L, LOWRANK_C = 64, 32
KERNELS_PER_ROUND_LOWRANK = 4  # one-pass verify_kernel, latent projection, finish (+ GEMV), latent fusion


def lowrank_flops(cfg: RoundConfig, R: int) -> int:
    """Flops of the low-rank conditioning: per conditioned row z = P m,
    t = B_c [z; u], rho = z + beta A_c t, [v; g_rho] = [W_v; W_g,rho] rho,
    plus W_g,e e once."""
    d, Lr, Cr = cfg.d, LOWRANK_L, LOWRANK_C
    per_row = 2 * (Lr * d + Cr * (Lr + d) + Lr * Cr + 2 * d * Lr)
    return R * per_row + 2 * d * d


def lowrank_bytes(cfg: RoundConfig, R: int) -> int:
    """Algorithmic bytes of the low-rank conditioning phase: the weights once
    (W_g's e columns dominate), the packed [m; u] rows read, e~ rows written."""
    es, d, Lr, Cr = cfg.elem_bytes, cfg.d, LOWRANK_L, LOWRANK_C
    weights = (Lr * d + Cr * (Lr + d) + Lr * Cr + d * Lr + d * (d + Lr)) * es
    return weights + R * 2 * d * es + R * d * es + d * es


def round_hbm_bytes(cfg: RoundConfig, R: int) -> int:
    """Algorithmic HBM bytes of one round: what must cross HBM at least once.

    Logits, draft tokens and outputs, the 2R conditioned hidden-state rows,
    the three weight matrices (5 d^2 elements), the mask embedding and e~.
    Packed intermediates are not counted (they can live in L2)."""
    es = cfg.elem_bytes
    B, K, V, d = cfg.B, cfg.K, cfg.V, cfg.d
    return (B * (K + 1) * V * es + B * K * 4 + B * (K + 1) * 4 + 3 * B * 4
            + 2 * R * d * es + 5 * d * d * es + d * es + B * K * d * es)


def round_is_fused(cfg: RoundConfig) -> bool:
    """Whether retrace_round takes the single-kernel path for this workload
    (bf16, d a multiple of 256, 16-byte aligned logits rows, K >= 2)."""
    return cfg.dtype == "bf16" and cfg.d % 256 == 0 and cfg.V % 8 == 0 and cfg.K >= 2


def run_gpu(args) -> dict | None:
    from paper_2608_29748_gb300 import binding as rt

    rank, local_rank, world = dist_env()
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    cfg = workload(args.config)
    peaks = load_peaks()

    x = make_round_inputs(cfg, device=dev, seed=shard_seed(42 + 1000 * cfg.seed_offset, rank))
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype, device=dev)
    out = rt.RoundBuffers(cfg.B, cfg.K, cfg.d, cfg.torch_dtype, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    fused = args.overlap and round_is_fused(cfg)
    if args.overlap and not fused:
        raise SystemExit("--overlap: the overlapped kernel does not cover this workload")
    if (args.lowrank or args.sampled) and (args.overlap or args.variant != "corrected"):
        raise SystemExit("--lowrank / --sampled run the corrected path alone")
    if args.lowrank and args.sampled:
        raise SystemExit("--lowrank and --sampled are separate paths")
    flags = VARIANT_FLAGS[args.variant] | (ROUND_OVERLAP_FLAG if fused else 0)
    if args.lowrank:
        from paper_2608_29748_gb300.workloads import make_lowrank_weights

        lw = make_lowrank_weights(cfg, device=dev, seed=shard_seed(77 + 1000 * cfg.seed_offset, rank))

        def round_fn(inputs, **kw):
            return rt.run_round_lowrank(inputs, lw, ws, out=out, **kw)
    elif args.sampled:
        from paper_2608_29748_gb300.workloads import make_sampled_inputs

        x.update(make_sampled_inputs(cfg, x["logits"], device=dev, seed=shard_seed(99 + 1000 * cfg.seed_offset, rank)))

        def round_fn(inputs, **kw):
            # a temperature-1 round: sampled verification, then the corrected, gated conditioning
            return rt.run_round_sampled(inputs, dict(inputs, temperature=x["temperature"], top_k=x["top_k"],
                                                     top_p=x["top_p"]), ws, out=out, **kw)
    else:
        def round_fn(inputs, **kw):
            return rt.run_round(inputs, ws, out=out, flags=flags, **kw)
    for _ in range(args.warmup):
        round_fn(x)
    torch.cuda.synchronize(dev)

    steps = args.steps
    # Two timed regions of K steps each.  The first gives `value`: one event
    # pair around each round, nothing inside it.  The second splits each round
    # into verification and conditioning with the library's phase events;
    # an event between two kernels keeps the second from starting early
    # (programmatic dependent launch), which costs about 11 us per round, so
    # those steps give the per-kernel durations of the rooflines only.
    outer = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(steps)]
    phase = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(steps)]
    for evs in outer + phase:
        for e in evs:
            e.record(stream)  # materialise the CUDA events before the timed regions
    torch.cuda.synchronize(dev)

    barrier(world)
    torch.cuda.synchronize(dev)
    with ClockSampler(local_rank) as clocks:
        t_wall0 = time.perf_counter()
        for i in range(steps):
            flush.fill_(i & 0xFF)  # L2 flush: a 256 MB write between timed steps
            outer[i][0].record(stream)
            round_fn(x)
            outer[i][1].record(stream)
        torch.cuda.synchronize(dev)
        t_wall = time.perf_counter() - t_wall0
        barrier(world)
        torch.cuda.synchronize(dev)
        for i in range(steps):
            flush.fill_(i & 0xFF)
            round_fn(x, phase_events=phase[i])
        torch.cuda.synchronize(dev)
    barrier(world)

    step_ms = [outer[i][0].elapsed_time(outer[i][1]) for i in range(steps)]
    phase_step_ms = [phase[i][0].elapsed_time(phase[i][3]) for i in range(steps)]
    verify_ms = [phase[i][0].elapsed_time(phase[i][1]) for i in range(steps)]
    cond_ms = [phase[i][1].elapsed_time(phase[i][3]) for i in range(steps)]
    round_s = sum(step_ms) / 1e3
    round_s_max = max_over_ranks(round_s, world, dev)
    value = aggregate_value(steps, world, round_s_max)

    n = out.n.cpu().numpy().astype(np.int64)
    accept = out.accept_len.cpu().numpy().astype(np.int64)
    R = int(n.sum())
    # verification: one pass, or passes over row windows plus one copy kernel
    # (a pass is one kernel greedy, top-k + finalize at temperature 1)
    windows = [0, cfg.K + 1] if fused else rt.retrace_verify_plan(cfg.B, cfg.K, cfg.V, cfg.torch_dtype)
    n_pass = len(windows) - 1
    verify_launches = n_pass * (2 if args.sampled else 1) + (1 if n_pass > 1 else 0)
    # one greedy pass that packs rows for the tensor-core projections hands the
    # decisions and copies to a second kernel when there are fewer sequences
    # than SMs (the finish kernel; the copy kernel at temperature 1)
    packs = cfg.dtype == "bf16" and (cfg.d % 64 == 0 if args.lowrank
                                     else cfg.d % 256 == 0 and (args.sampled or args.variant in ("corrected", "raw")))
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    if n_pass == 1 and not fused and packs and cfg.B < sms:
        verify_launches += 1
    # conditioning launches of the greedy and temperature-1 rounds, by path
    rows = (cfg.B * (cfg.K - 1) + 15) // 16 * 16
    small_r = 0 < rows <= 1024 and (2 * cfg.d // 128) * ((rows + 255) // 256) <= 256
    if cfg.dtype != "bf16" or cfg.d % 256:
        cond_launches = 3  # correction, gate bias, gate (FFMA)
    elif small_r and rows <= 256:
        # split-K clusters: correction, gate-bias GEMV, gate (raw: GEMV, gate)
        cond_launches = 3 if args.variant == "corrected" else 2
    elif small_r:
        cond_launches = 4 if args.variant == "corrected" else 3  # GEMM + reduction each; raw: GEMV, GEMM, reduction
    else:
        cond_launches = 1  # cond_pair_kernel
    step_avg_s = statistics.mean(step_ms) / 1e3
    cflops = (lowrank_flops(cfg, R) if args.lowrank
              else conditioning_flops(cfg, R, dense_e=False, variant=args.variant))
    status_flags = ws.check()
    if fused:
        # One kernel does the whole round: its floor is the larger of the HBM
        # time of its algorithmic bytes and the tensor time of its flops.
        hbytes = round_hbm_bytes(cfg, R)
        t_hbm = hbytes / (peaks["hbm_gbs"] * 1e9)
        t_tc = cflops / (peaks["bf16_tflops_sustained"] * 1e12)
        hbm_bound = t_hbm >= t_tc
        roofline = {
            "kernel": "cond_kernel<FUSED> (verification + both projections, one persistent launch per round)",
            "bound": "hbm" if hbm_bound else "tensor",
            "achieved": round(hbytes / step_avg_s / 1e9, 1) if hbm_bound else round(cflops / step_avg_s / 1e12, 2),
            "peak": peaks["hbm_gbs"] if hbm_bound else peaks["bf16_tflops_sustained"],
            "unit": "GB/s" if hbm_bound else "TFLOP/s",
            "frac": round(max(t_hbm, t_tc) / step_avg_s, 4),
            "peak_source": peaks["source"] + (" HBM copy bandwidth" if hbm_bound else " sustained bf16 (cuBLAS)"),
            "algorithmic_bytes": hbytes,
            "algorithmic_flops": cflops,
            "floor_us": {"hbm": round(t_hbm * 1e6, 1), "tensor": round(t_tc * 1e6, 1)},
            "avg_launch_us": round(step_avg_s * 1e6, 2),
            "traffic": measured_traffic("overlapped", cfg.name, args.variant),
            "traffic_source": "ncu dram read+write of the round's kernel on this workload",
        }
        line_extra = {"hbm_view": {"achieved_gbs": round(hbytes / step_avg_s / 1e9, 1),
                                   "frac": round(t_hbm / step_avg_s, 4)},
                      "tensor_view": {"achieved_tflops": round(cflops / step_avg_s / 1e12, 2),
                                      "frac": round(t_tc / step_avg_s, 4)}}
    else:
        packs_rows = cfg.dtype == "bf16" and cfg.d % 256 == 0  # tensor-core path: verify packs the rows
        vbytes = verify_bytes(cfg, n, packs_rows and args.variant in ("corrected", "raw"), args.variant, accept)
        rbytes = vbytes - needed_logits_bytes(cfg, accept) + read_logits_bytes(cfg, accept, windows)
        v_avg_s = statistics.mean(verify_ms) / 1e3
        c_avg_s = statistics.mean(cond_ms) / 1e3
        c_tflops = cflops / c_avg_s / 1e12
        if args.sampled:  # drafter rows 0..min(A_b, K-1) and the uniforms are needed too
            d_needed = int(np.sum(np.minimum(accept + 1, cfg.K))) * cfg.V * cfg.elem_bytes
            d_rows = sum(int(np.sum(accept >= windows[k])) * max(0, min(windows[k + 1], cfg.K) - windows[k])
                         for k in range(n_pass))
            vbytes += d_needed + cfg.B * (cfg.K + 1) * 4
            rbytes += d_rows * cfg.V * cfg.elem_bytes + cfg.B * (cfg.K + 1) * 4
        v_gbs = vbytes / v_avg_s / 1e9
        copies = (" + verify_copy_kernel (copy of unconditioned rows + row packing)" if args.sampled else
                  " (keys only) + verify_finish_kernel (decisions, copy of unconditioned rows + row packing)")
        passes = "sampled_topk_kernel + sampled_finalize_kernel" if args.sampled else "verify_kernel"
        if n_pass > 1:
            finish = (" + verify_finish_kernel (decisions of the last window, copy of unconditioned rows + row "
                      "packing)")
            v_kernel = f"{passes} x{n_pass} passes over row windows {windows}{finish}"
        elif verify_launches > (2 if args.sampled else 1):
            v_kernel = f"{passes} (one pass){copies}"
        else:
            v_kernel = f"{passes} (one pass; the finalisers copy unconditioned rows and pack rows)"
        v_roof = {
            "kernel": v_kernel,
            "bound": "hbm",
            "achieved": round(v_gbs, 1),
            "peak": peaks["hbm_gbs"],
            "unit": "GB/s",
            "frac": round(v_gbs / peaks["hbm_gbs"], 4),
            "peak_source": peaks["source"] + " HBM copy bandwidth",
            "algorithmic_bytes": vbytes,
            "algorithmic_bytes_note": "logits rows 0..A_b of each sequence (what the outputs depend on), tokens, "
                                      "row copies and packing",
            "bytes_streamed": rbytes,
            "streamed_frac": round(rbytes / v_avg_s / 1e9 / peaks["hbm_gbs"], 4),
            "launches": verify_launches,
            "avg_launch_us": round(v_avg_s * 1e6, 2),
            "traffic": None if args.sampled else measured_traffic("verify", cfg.name, args.variant),
            "traffic_source": "ncu dram read+write of the verification kernels (passes + finishing or copy "
                              "kernel) of one round on this workload",
        }
        if args.variant in ("overwrite", "none"):
            v_roof["kernel"] = v_roof["kernel"].replace("copy of unconditioned rows + row packing",
                                                        "every row of e~ copied")
        if args.sampled:
            v_roof["kernel"] = (f"sampled_topk_kernel + sampled_finalize_kernel x{n_pass} passes over row windows "
                                f"{windows} (top-k of the window's target and drafter rows, accept tests, draw)"
                                + (" + verify_copy_kernel (copy of unconditioned rows + row packing)"
                                   if n_pass > 1 else " (+ copy of unconditioned rows + row packing)"))
            v_roof["traffic"] = None
        c_roof = None
        if args.lowrank:
            cbytes = lowrank_bytes(cfg, R)
            c_roof = {
                "kernel": "low-rank conditioning: latent projection (tcgen05, split-K), finish (rho, + the "
                          "gate-bias GEMV), latent fusion (tcgen05, persistent)",
                "bound": "hbm",
                "achieved": round(cbytes / c_avg_s / 1e9, 1),
                "peak": peaks["hbm_gbs"],
                "unit": "GB/s",
                "frac": round(cbytes / c_avg_s / 1e9 / peaks["hbm_gbs"], 4),
                "peak_source": peaks["source"] + " HBM copy bandwidth",
                "algorithmic_bytes": cbytes,
                "algorithmic_flops": cflops,
                "avg_launch_us": round(c_avg_s * 1e6, 2),
                "traffic": None,
            }
        elif cflops:
            c_roof = {
                "kernel": ("cond_pair_kernel: correction + gated-fusion projections (+ gate-bias GEMV), one persistent "
                           "launch on CTA pairs (tcgen05.mma.cta_group::2)"),
                "bound": "tensor",
                "achieved": round(c_tflops, 2),
                "peak": peaks["bf16_tflops"],
                "unit": "TFLOP/s",
                "frac": round(c_tflops / peaks["bf16_tflops"], 4),
                "peak_source": peaks["source"] + " burst bf16 (cuBLAS); the kernel runs at full SM clock",
                "frac_of_sustained": round(c_tflops / peaks["bf16_tflops_sustained"], 4),
                "algorithmic_flops": cflops,
                "avg_launch_us": round(c_avg_s * 1e6, 2),
                "traffic": None if args.sampled else measured_traffic("conditioning", cfg.name, args.variant),
                "traffic_source": "ncu dram read+write of one launch on this workload",
            }
            if cfg.dtype != "bf16" or cfg.d % 256:
                # fp32 (no TF32) or shapes the tensor-core kernels do not take: plain FFMA
                props = torch.cuda.get_device_properties(dev)
                max_mhz = (clocks.summary() or {}).get("sm_max_mhz") or 2070.0
                ffma_peak = props.multi_processor_count * 128 * 2 * max_mhz * 1e6 / 1e12
                c_roof.update({
                    "kernel": ("FFMA path: simt_rows_correct_kernel, gate_bias_kernel, simt_rows_gate_kernel (a warp per "
                               "feature)" if cfg.B * (cfg.K - 1) <= 32 else
                               "FFMA path: simt_correct_kernel, gate_bias_kernel, simt_gate_kernel"),
                    "bound": "alu", "peak": round(ffma_peak, 1), "frac": round(c_tflops / ffma_peak, 4),
                    "peak_source": "derived: SMs x 128 FP32 lanes x 2 flop per FMA x maximum SM clock",
                    "frac_of_sustained": None, "traffic": None})
            elif small_r:
                # weights streamed once dominate: HBM-bound at these row counts
                es, d = cfg.elem_bytes, cfg.d
                cbytes = 5 * d * d * es + R * (2 * d + d + d) * es + R * d * 2
                c_roof.update({
                    "kernel": ("small-R GEMMs: swap_cluster_kernel (tcgen05, weights as the 128-row side, split-K "
                               "over a cluster whose partials are summed in distributed shared memory) for each "
                               "projection, swap_gemv_kernel beside the correction" if rows <= 256 else
                               "small-R GEMMs: swap_gemm_kernel (tcgen05, weights as the 128-row side, split-K) for "
                               "each projection, each followed by its reduction kernel"),
                    "bound": "hbm", "achieved": round(cbytes / c_avg_s / 1e9, 1), "peak": peaks["hbm_gbs"],
                    "unit": "GB/s", "frac": round(cbytes / c_avg_s / 1e9 / peaks["hbm_gbs"], 4),
                    "peak_source": peaks["source"] + " HBM copy bandwidth",
                    "algorithmic_bytes": cbytes,
                    "algorithmic_bytes_note": "W_c, W_v, W_g once; packed [m; u] rows read, r written and read, "
                                              "e~ rows written",
                    "achieved_tflops": round(c_tflops, 3), "frac_of_sustained": None, "traffic": None})
        # `roofline` is the kernel that takes the larger share of the round
        roofline = c_roof if (c_roof and c_avg_s > v_avg_s) else v_roof
        line_extra = {"roofline_verify": v_roof, "roofline_conditioning": c_roof}

    # ---- end to end through the public API with host buffers ----
    names = ["logits", "draft", "hD", "hT"] + (["draft_logits", "uniforms"] if args.sampled else [])
    e2e = run_e2e(cfg, x, dev, min(steps, args.e2e_steps), world, round_fn, names) if args.e2e_steps > 0 else None

    line = {
        "metric": METRIC,
        "value": round(value, 3),
        "unit": UNIT,
        "n_gpus": world,
        "steps": steps,
        "warmup": args.warmup,
        "ms_per_step": round(statistics.mean(step_ms), 4),
        "ms_per_step_with_phase_events": round(statistics.mean(phase_step_ms), 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16" if cfg.dtype == "bf16" else "f32",
        "data": "synthetic (seeded; Qwen3-8B / DFlash-b16 shapes, random-init fusion weights)",
        "config": {
            "workload": f"{cfg.name}: B={cfg.B} K={cfg.K} V={cfg.V} d={cfg.d} {cfg.dtype}, "
                        f"prefix {cfg.prefix}({cfg.prefix_p or ''}) capped at K",
            "B": cfg.B, "K": cfg.K, "V": cfg.V, "d": cfg.d,
            "conditioned_rows_R": R,
            "l2": "flushed before every timed step (256 MB write, outside the per-step events)",
            "parallelism": f"replicas x{world} (batch-sharded, no collective)",
            "variant": ("low-rank (rank-64 latents, rank-32 correction)" if args.lowrank
                        else f"temperature {x['temperature']}, top_k {x['top_k']}, top_p {x['top_p']} "
                             "(speculative sampling)" if args.sampled else args.variant),
            "verify_windows": windows,
            "round_kernel": ("overlapped (one persistent launch)" if fused
                             else f"verify ({verify_launches} launches), latent projection, finish + GEMV, "
                                  "latent fusion" if args.lowrank
                             else f"verify ({verify_launches} launches: sampled top-k + finalize per pass), "
                                  "projections" if args.sampled
                             else f"verify ({verify_launches} launches), projections" if cflops
                             else f"verify ({verify_launches} launches)"),
        },
        "roofline": roofline,
        **line_extra,
        "e2e": e2e,
        "gpu_launches": (KERNELS_PER_ROUND_FUSED if fused
                         else KERNELS_PER_ROUND_LOWRANK - 1 + verify_launches if args.lowrank
                         else verify_launches + cond_launches if (args.sampled or cflops)
                         else verify_launches) * steps,
        "wall_s_timed_region": round(t_wall, 4),
        "device_status_flags": status_flags,
        "impl": "ours",
    }
    cs = clocks.summary()
    line["clocks"] = cs
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(cfg, args)
    return line if rank == 0 else None


def run_e2e(cfg, x, dev, steps, world, round_fn, names) -> dict:
    """Rounds/s with the step's inputs in pinned host memory and the outputs read back."""
    host = {k: x[k].cpu().pin_memory() for k in names}
    dev_in = {k: torch.empty_like(x[k]) for k in names}
    rest = {k: x[k] for k in ("e", "Wc", "Wv", "Wg", "beta", "cfg")}  # model parameters stay resident
    out = round_fn(x)  # the round's output buffers
    out_host = {k: torch.empty(getattr(out, k).shape, dtype=getattr(out, k).dtype).pin_memory()
                for k in ("accept_len", "committed", "bonus", "n", "e_out")}
    stream = torch.cuda.current_stream(dev)

    def step():
        for k in names:
            dev_in[k].copy_(host[k], non_blocking=True)
        round_fn({**dev_in, **rest})
        for k, h in out_host.items():
            h.copy_(getattr(out, k), non_blocking=True)

    step()
    torch.cuda.synchronize(dev)
    barrier(world)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for _ in range(steps):
        step()
    end.record(stream)
    torch.cuda.synchronize(dev)
    secs = max_over_ranks(start.elapsed_time(end) / 1e3, world, dev)
    h2d = sum(h.numel() * h.element_size() for h in host.values())
    d2h = sum(h.numel() * h.element_size() for h in out_host.values())
    return {"value": round(aggregate_value(steps, world, secs), 3), "unit": UNIT,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": steps}


CPU_BASELINE_SECONDS = 10.0  # the oracle's sample is repeated until it has run this long


def cpu_baseline(cfg: RoundConfig, args) -> dict:
    host = prepare_oracle_sample(cfg, args.cpu_sample, seed=1234, lowrank=args.lowrank, sampled=args.sampled)
    times = []
    while sum(times) < CPU_BASELINE_SECONDS and len(times) < 200:
        times.append(time_oracle(host, args.variant))
    secs = sum(times) / len(times)
    rounds = host["B"] / cfg.B
    return {"value": round(rounds / secs, 6), "unit": UNIT, "cores": cpu_threads(), "kind": "oracle",
            "sample": f"{host['B']} of {cfg.B} sequences of {cfg.name}, full-size weights, run {len(times)} times "
                      f"({sum(times):.1f} s of CPU work); one round of the sample took {secs:.2f} s on average, "
                      f"scaled by {host['B']}/{cfg.B} to rounds/s"}


# ---------------------------------------------------------------------------
# reference arm: the CPU oracle on the same workload
# ---------------------------------------------------------------------------


def run_reference(args) -> dict | None:
    rank, _, world = dist_env()
    if rank != 0:
        return None
    cfg = workload(args.config)
    host = prepare_oracle_sample(cfg, args.ref_sample, seed=500, lowrank=args.lowrank, sampled=args.sampled)
    for _ in range(min(args.warmup, 1)):
        time_oracle(host, args.variant)
    total = sum(time_oracle(host, args.variant) for _ in range(args.steps))
    value = args.steps * (host["B"] / cfg.B) / total
    return {
        "metric": METRIC, "value": round(value, 6), "unit": UNIT, "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(1e3 * total / args.steps, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": f"{cfg.name}: B={cfg.B} K={cfg.K} V={cfg.V} d={cfg.d} {cfg.dtype}",
                   "sample_per_step": f"{args.ref_sample} of {cfg.B} sequences (full-size weights)",
                   "variant": args.variant},
        "impl": "reference",
        "cpu_baseline": {"value": round(value, 6), "unit": UNIT, "cores": cpu_threads(), "kind": "oracle",
                         "sample": f"{args.ref_sample} of {cfg.B} sequences per step, {args.steps} steps, "
                                   f"scaled by {args.ref_sample}/{cfg.B} to rounds/s"},
        "e2e": {"value": round(value, 6), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def run_sweep(args) -> None:
    """Every workload (configs 1-5): verification alone and the whole round,
    the median of max(steps, 50) CUDA-event timings after warm-up, cold (a
    256 MB L2 flush before every call) and warm (back to back, so whatever
    fits stays in L2), plus CUDA-graph replay of the round for B <= 8.  Also
    the bytes verification needs at least, sum_b (A_b + 1) V s (the rows up to
    the first mismatch), against the bytes its schedule streams (every row in
    one pass, or the row windows of the still-matching sequences).  One JSON
    line per workload; an extra report, not the benchmark line."""
    from paper_2608_29748_gb300 import binding as rt

    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    peaks = load_peaks()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    iters = max(args.steps, 50)

    def timed(fn, cold: bool) -> float:
        for _ in range(max(args.warmup, 3)):
            fn()
        torch.cuda.synchronize(dev)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(iters)]
        for i in range(iters):
            if cold:
                flush.fill_(i & 0xFF)
            ev[i][0].record()
            fn()
            ev[i][1].record()
        torch.cuda.synchronize(dev)
        return statistics.median(a.elapsed_time(b) for a, b in ev) * 1e3  # µs

    for cid in sorted(CONFIGS):
        cfg = CONFIGS[cid]
        x = make_round_inputs(cfg, device=dev)
        ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype, device=dev)
        out = rt.RoundBuffers(cfg.B, cfg.K, cfg.d, cfg.torch_dtype, device=dev)

        def verify():
            rt.retrace_verify(x["logits"], x["draft"], out.accept_len, out.committed, out.bonus, ws)

        def round_():
            rt.run_round(x, ws, out=out)

        v = {"cold": timed(verify, True), "warm": timed(verify, False)}
        r = {"cold": timed(round_, True), "warm": timed(round_, False)}
        graph = None
        if cfg.B <= 8:
            s = torch.cuda.Stream(dev)
            s.wait_stream(torch.cuda.current_stream(dev))
            with torch.cuda.stream(s):
                rt.run_round(x, ws, out=out, stream=s)
            torch.cuda.current_stream(dev).wait_stream(s)
            torch.cuda.synchronize(dev)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=s):
                rt.run_round(x, ws, out=out, stream=s)
            graph = {"cold": timed(g.replay, True), "warm": timed(g.replay, False)}
        round_()
        torch.cuda.synchronize(dev)
        A = out.accept_len.cpu().numpy().astype(np.int64)
        n = out.n.cpu().numpy().astype(np.int64)
        windows = rt.retrace_verify_plan(cfg.B, cfg.K, cfg.V, cfg.torch_dtype)
        logits = read_logits_bytes(cfg, A, windows)  # what the schedule streams
        needed = needed_logits_bytes(cfg, A)
        line = {
            "config": cid, "workload": cfg.name, "B": cfg.B, "K": cfg.K, "V": cfg.V, "d": cfg.d,
            "dtype": cfg.dtype, "conditioned_rows_R": int(n.sum()), "iters": iters, "statistic": "median",
            "verify_windows": windows,
            "verify_us": {k: round(t, 2) for k, t in v.items()},
            "streamed_gbs": {k: round(logits / t / 1e3, 1) for k, t in v.items()},
            "logits_frac_of_hbm": {k: round(logits / t / 1e3 / peaks["hbm_gbs"], 4) for k, t in v.items()},
            "needed_gbs": {k: round(needed / t / 1e3, 1) for k, t in v.items()},
            "round_us": {k: round(t, 2) for k, t in r.items()},
            "rounds_per_s": {k: round(1e6 / t, 1) for k, t in r.items()},
            "graph_round_us": None if graph is None else {k: round(t, 2) for k, t in graph.items()},
            "logits_bytes_streamed": logits,
            "needed_bytes_rows_to_first_mismatch": needed,
            "needed_us_at_hbm_peak": round(needed / (peaks["hbm_gbs"] * 1e3), 2),
            "hbm_peak_gbs": peaks["hbm_gbs"], "peak_source": peaks["source"],
        }
        print(json.dumps(line), flush=True)
        del x, ws, out
        torch.cuda.empty_cache()


def workload(name: str) -> RoundConfig:
    return PROFILE_CONFIG if name == "profile" else CONFIGS[int(name)]


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="5", choices=[str(k) for k in sorted(CONFIGS)] + ["profile"],
                    help="workload 1-5, or 'profile' (B=128 half batch for profiler captures)")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--cpu-sample", type=int, default=32, help="sequences in the CPU-baseline sample")
    ap.add_argument("--ref-sample", type=int, default=2, help="sequences per step in the reference arm")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--overlap", action="store_true",
                    help="time the overlapped single-kernel round (RETRACE_ROUND_OVERLAP)")
    ap.add_argument("--sampled", action="store_true",
                    help="time a temperature-1 round (retrace_round_sampled)")
    ap.add_argument("--lowrank", action="store_true",
                    help="time the low-rank conditioning path (retrace_round_lowrank)")
    ap.add_argument("--variant", choices=sorted(VARIANT_FLAGS), default="corrected",
                    help="conditioning variant of the component ablation (default: the method)")
    ap.add_argument("--sweep", action="store_true",
                    help="report every workload (1-5): verification and round, cold and warm medians, "
                         "graph replay for B <= 8; one JSON line each (not the benchmark line)")
    return ap.parse_args(argv)


def main(argv=None) -> None:
    args = parse_args(argv)
    if args.warmup < 3 and args.impl == "ours":
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)
    if args.sweep:
        run_sweep(args)
        return
    line = run_reference(args) if args.impl == "reference" else run_gpu(args)
    if line is not None:
        print(json.dumps(line), flush=True)
    _, _, world = dist_env()
    if world > 1 and args.impl == "ours":
        import torch.distributed as dist

        dist.destroy_process_group()


if __name__ == "__main__":
    main()

"""Throughput of the grid iteration: G-D pair evaluations per second and grid iterations per
second on one GB300, with the roofline fraction of the dominant kernel, an end-to-end number
through the C ABI with host buffers, and the CPU oracle timed on a bounded sample.

Workload: 12x12 toroidal grid (144 cells, 720 neighbourhood slots, 3600 G-D pairs per
iteration), MLP G (64-256-256-784) and D (784-256-256-1), bf16 operands with fp32 accumulation
and fp32 Adam masters, minibatch 100, real data from a seeded 10-blob 784-dim pool. One step is
one full grid iteration (minibatch draw, all-pairs evaluation, fitness, selection, backward and
Adam of every cell's new centre pair).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--train-steps S] [--mixture] [--stale-neighbors] [--dcgan]

With --train-steps S > 1 every iteration trains each cell's new centre pair S times (the later
steps on fresh minibatches); the default S = 1 is the headline workload. --mixture adds the
generator-mixture ES-(1+1) step (Gaussian-kernel MMD score) to every evaluation;
--stale-neighbors runs the asynchronous schedule (neighbours one iteration late). --dcgan
times the 3x3 DCGAN configuration (width 64, z = 100, B = 128, bf16) instead of the MLP.

With N > 1 (torchrun, one process per GPU) every rank runs its own 12x12 grid (replicas: the
per-GPU work is fixed, scaling "weak"); value = all ranks' pairs / the slowest rank's time.
"""

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

ROWS, COLS, BATCH = 12, 12, 100
Z_DIM, HIDDEN, X_DIM = 64, 256, 784
POOL_N, SEED = 60000, 1811
CELLS = ROWS * COLS
PAIRS = 25 * CELLS
METRIC = "G-D pair evals/sec and grid iterations/sec on 1 GB300; % of bf16 tensor peak"
UNIT = "pair-evals/s"
WORKLOAD = "12x12 torus MLP G/D bf16 B=100 (3600 pairs/iter)"

# Algorithmic work per iteration (no padding, no recomputation):
#   evaluation: generator slots 5 B rows x (z*h + h*h + h*x) MACs per cell; discriminator slots
#   5 * 6B rows x (x*h + h*h + h) MACs per cell.
G_MAC_ROW = Z_DIM * HIDDEN + HIDDEN * HIDDEN + HIDDEN * X_DIM            # 282,624
D_MAC_ROW = X_DIM * HIDDEN + HIDDEN * HIDDEN + HIDDEN                    # 266,496
PG = HIDDEN * Z_DIM + HIDDEN + HIDDEN * HIDDEN + HIDDEN + X_DIM * HIDDEN + X_DIM
PD = HIDDEN * X_DIM + HIDDEN + HIDDEN * HIDDEN + HIDDEN + HIDDEN + 1
# The backward kernel applies Adam to the weight matrices (G: W1, W2, W3; D: W1, W2) in its
# epilogue, and to the remaining parameters (both networks' biases, D's output layer) once a
# cell's tiles are done: per parameter it reads the old w, m, v (12 B) and writes the new w, m,
# v and the bf16 copy (14 B), plus the fp32 gradient of the remaining ones (4 B). Its other algorithmic reads: the bf16 weights of the four matrices the
# delta chain multiplies by (D: W2, W1; G: W3, W2) and the stored forward activations
# (J2 3B x h, TG1 2B x h, TX 2B x x, TH1 and TH2 B x h, Z B x z), all bf16.
W_FUSED = (Z_DIM * HIDDEN + HIDDEN * HIDDEN + X_DIM * HIDDEN) + (HIDDEN * X_DIM + HIDDEN * HIDDEN)
BWD_ACT = (3 * BATCH * HIDDEN + 2 * BATCH * HIDDEN + 2 * BATCH * X_DIM + 2 * BATCH * HIDDEN
           + BATCH * Z_DIM)
W_RANGES = (HIDDEN + HIDDEN + X_DIM) + (HIDDEN + HIDDEN + HIDDEN + 1)  # biases, D's W3 and b3


def _derive():
    """The per-iteration work of a ROWS x COLS torus (module globals, so that --grid can set a
    smaller torus for kernel captures)."""
    global CELLS, PAIRS, EVAL_G_FLOP, EVAL_D_FLOP, TRAIN_FWD_FLOP, TRAIN_BWD_FLOP, MIX_FLOP
    global TRAIN_BWD_BYTES
    CELLS = ROWS * COLS
    PAIRS = 25 * CELLS
    EVAL_G_FLOP = 2 * CELLS * 5 * BATCH * G_MAC_ROW
    EVAL_D_FLOP = 2 * CELLS * 30 * BATCH * D_MAC_ROW
    # Training: forward of the selected pair (G layers 1-2 on B rows, D on 2B rows), backward.
    TRAIN_FWD_FLOP = (2 * CELLS * BATCH * (Z_DIM * HIDDEN + HIDDEN * HIDDEN)
                      + 2 * CELLS * 2 * BATCH * D_MAC_ROW)
    TRAIN_BWD_FLOP = 2 * CELLS * BATCH * 1479936
    # Mixture step (--mixture): the Gram matrix of every cell's 6B evaluation rows.
    MIX_FLOP = 2 * CELLS * (6 * BATCH) ** 2 * X_DIM
    TRAIN_BWD_BYTES = CELLS * (26 * W_FUSED + 30 * W_RANGES
                               + 2 * (2 * HIDDEN * HIDDEN + 2 * X_DIM * HIDDEN) + 2 * BWD_ACT)


_derive()

# DRAM bytes (read + write) per phase of one iteration, summed over the phase's kernels: not
# measured by this script but taken from ncu captures (dram__bytes_read.sum +
# dram__bytes_write.sum) of these same kernels, each with the summary it comes from. A phase
# whose kernels changed after its capture has no entry (null traffic).
PHASE_TRAFFIC = {
    "train_bwd": (2198.7e6, "profiles/k_bwd_cells_fused_adam_12x12_bf16.md"),
    "d_fwd": (236.6e6, "profiles/k_mlp_fwd_pair_eval_12x12_bf16.md"),
    "g_fwd": (146.4e6, "profiles/k_mlp_fwd_pair_eval_12x12_bf16.md"),
    "batch": (21.2e6, "profiles/launches_12x12_bf16_iteration.md (earlier DRAM capture)"),
    "fitness": (1.8e6, "profiles/launches_12x12_bf16_iteration.md (earlier DRAM capture)"),
}


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d.get("hbm_gbs", 6800.0), d.get("bf16_tflops", 1900.0), \
            d.get("bf16_tflops_sustained", 1700.0), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during a timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()
        return False

    def summary(self):
        rows = [r.split(", ") for r in (self.out or "").strip().splitlines() if r.strip()]
        rows = [r for r in rows if len(r) >= 9]
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].strip() == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


def allreduce_max(dist, x):
    """Largest value of x over the ranks (CPU tensors under gloo, CUDA tensors under NCCL)."""
    import torch
    if dist is None:
        return float(x)
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate(ms_per_rank_max, steps, world):
    """(ms per step, grid iterations / s, pair evaluations / s) of the whole job from the
    slowest rank's time: every rank runs its own 12x12 grid, so the job's pairs are world x."""
    ms_step = ms_per_rank_max / steps
    iters_s = 1000.0 / ms_step
    return ms_step, iters_s * world, PAIRS * world * iters_s


def _dist():
    n = int(os.environ.get("WORLD_SIZE", "1"))
    if n > 1:
        import torch.distributed as dist
        if not dist.is_initialized():
            dist.init_process_group("nccl" if os.environ.get("LIPZ_BENCH_GLOO") is None else "gloo")
        return dist, dist.get_rank(), n
    return None, 0, 1


def run_ours(args):
    import numpy as np
    import torch

    dist, rank, world = _dist()
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    import __graft_entry__
    __graft_entry__.build()
    import lipz_synth
    import paper_1811_12843_gb300 as L

    pool = lipz_synth.blob_pool(SEED, n=POOL_N, dim=X_DIM)
    g = L.Grid(ROWS, COLS, seed=SEED + rank, precision="bf16", batch=BATCH,
               train_steps=args.train_steps, mixture=1 if args.mixture else 0,
               stale_neighbors=1 if args.stale_neighbors else 0)
    g.set_data(pool)
    stream = torch.cuda.Stream()
    g.set_stream(stream.cuda_stream)

    def barrier():
        torch.cuda.synchronize()
        if dist:
            dist.barrier()

    # warm-up
    for _ in range(args.warmup):
        L.lipz_iterate(g.h, 1)
    g.synchronize()
    L.lipz_profile_read(g.h)  # reset counters

    # ---- timed region: K grid iterations on the grid's stream (device time)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    with Clocks(local) as clk:
        e0.record(stream)
        for _ in range(args.steps):
            L.lipz_iterate(g.h, 1)
        e1.record(stream)
        g.synchronize()
    barrier()
    ms = e0.elapsed_time(e1)
    prof0 = L.lipz_profile_read(g.h)
    launches = sum(v[2] for v in prof0.values())
    ms_step, iters_total, value = aggregate(allreduce_max(dist, ms), args.steps, world)

    # ---- per-phase device time (separate pass with phase events on the same stream)
    phase_ms = {k: float("nan") for k in L.PHASES}
    if not args.no_phases:
        L.lipz_profile_enable(g.h, True)
        for _ in range(args.steps):
            L.lipz_iterate(g.h, 1)
        prof = L.lipz_profile_read(g.h)
        L.lipz_profile_enable(g.h, False)
        phase_ms = {k: v[0] / max(v[1], 1) for k, v in prof.items()}

    # ---- end to end through the public API: pinned host minibatches in, fitness out
    if args.no_e2e:
        e2e_value = None
    else:
        e2e_value = _e2e(args, L, g, torch, dist, world)
    h2d = CELLS * BATCH * X_DIM * 4
    d2h = 2 * CELLS * 5 * 4 + 8 * 4  # fitnesses and the eight device status words, one copy
    if args.no_phases:
        roof = None
    else:
        roof = _roofline(phase_ms)
    if rank != 0:
        return None
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded 10-blob 784-dim pool standing in for MNIST)",
        "config": {"workload": _workload(args),
                   "rows": ROWS, "cols": COLS, "global_batch": BATCH,
                   "train_steps": args.train_steps,
                   "pairs_per_iter": PAIRS, "parallelism": "replicas" if world > 1 else "single",
                   "l2": "inputs larger than L2 (population 2.2 GB + pool 188 MB per iteration)"},
        "grid_iterations_per_sec": iters_total,
        "pair_evals_per_sec_eval_only": PAIRS * world * 1000.0 /
        (phase_ms["batch"] + phase_ms["g_fwd"] + phase_ms["d_fwd"] + phase_ms["fitness"]),
        "phase_ms": phase_ms,
        "roofline": roof,
        "phase_rooflines": None if args.no_phases else _phase_roofs(phase_ms),
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": launches,
        "clocks": clk.summary(),
    }
    if (world == 1 and not args.no_cpu_baseline and args.train_steps == 1 and not args.mixture
            and not args.stale_neighbors):
        line["cpu_baseline"] = cpu_baseline(args.cpu_seconds, args.cpu_seconds_single)
    return line


def _e2e(args, L, g, torch, dist, world):
    import lipz_synth
    nbuf = 2
    xs = [torch.from_numpy(lipz_synth.host_batch(SEED + 7 + i, CELLS, BATCH, X_DIM)).pin_memory()
          for i in range(nbuf)]
    # two sets of pinned result buffers: a call's fitnesses land while the next call runs
    fit = [(torch.zeros((CELLS, 5), dtype=torch.float32).pin_memory(),
            torch.zeros((CELLS, 5), dtype=torch.float32).pin_memory()) for _ in range(2)]
    for i in range(2):
        L.lipz_iterate_batch(g.h, xs[i % nbuf], fit[0][0], fit[0][1])
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    # every step's upload and fitness read-back is inside the timed region: the first upload
    # with its own call, each later one issued by the call before it, which overlaps it with
    # that iteration's compute; lipz_iterate_batch_async returns once the previous call's
    # iteration (and its fitness copy) is complete, and lipz_synchronize completes the last
    t0 = time.perf_counter()
    for i in range(args.steps):
        nxt = xs[(i + 1) % nbuf] if i + 1 < args.steps else None
        L.lipz_iterate_batch_async(g.h, xs[i % nbuf], nxt, fit[i % 2][0], fit[i % 2][1])
    L.lipz_synchronize(g.h)
    e2e_s = allreduce_max(dist, time.perf_counter() - t0)
    return PAIRS * world * args.steps / e2e_s


def _phase_roofs(phase_ms):
    """Roofline of every heavy phase: algorithmic work / device time against the measured peak."""
    hbm, tf_burst, tf_sus, peak_kind = _peaks()
    work = {"g_fwd": ("tensor", EVAL_G_FLOP, "generator evaluation forward (all 720 slots, 3 fused layers)"),
            "d_fwd": ("tensor", EVAL_D_FLOP,
                      "discriminator evaluation forward (all 720 slots, 3 fused layers + logit)"),
            "train_fwd": ("tensor", TRAIN_FWD_FLOP, "forward of every cell's selected pair"),
            "mixture": ("tensor", MIX_FLOP, "mixture score: Gram of every cell's 6B evaluation "
                        "rows with the Gaussian kernel and block sums fused, plus the ES step"),
            "train_bwd": ("hbm", TRAIN_BWD_BYTES,
                          "backward of every cell's selected pair with Adam + replacement of "
                          "the weight matrices fused in (%.1f GFLOP)" % (TRAIN_BWD_FLOP / 1e9))}
    out = {}
    for ph, (bound, units, what) in work.items():
        t = phase_ms.get(ph)
        if not t or t != t:
            continue
        if bound == "hbm":
            ach, peak, unit = units / (t * 1e-3) / 1e9, hbm, "GB/s"
            src = peak_kind + " HBM copy"
        else:
            # the timed region lasts milliseconds, not seconds: the burst rate applies
            ach, peak, unit = units / (t * 1e-3) / 1e12, tf_burst, "TFLOP/s"
            src = peak_kind + " burst bf16 (cuBLAS)"
        tr, tr_src = PHASE_TRAFFIC.get(ph, (None, None))
        out[ph] = {"bound": bound, "achieved": ach, "peak": peak, "unit": unit, "frac": ach / peak,
                   "traffic": tr, "traffic_source": tr_src,
                   "kernel": what, "peak_source": src,
                   ("algorithmic_bytes" if bound == "hbm" else "algorithmic_flop"): units}
    return out


def _roofline(phase_ms):
    """Roofline of the phase with the largest device time."""
    roofs = _phase_roofs(phase_ms)
    dom = max(roofs, key=lambda k: phase_ms[k])
    r = dict(roofs[dom])
    r["phase"] = dom
    return r


def _oracle_sample(seconds, max_cells=None, train_steps=1, mixture=False, stale=False):
    """Run the oracle's full iteration cell by cell on the 12x12 workload until ``seconds`` of
    CPU work are spent; return (cells done, elapsed seconds). With ``train_steps`` K > 1 each
    cell's pair then takes K - 1 more steps on fresh minibatches; with ``mixture`` each cell also
    takes its mixture ES step."""
    import numpy as np
    import lipz_synth
    from oracle import lipz_oracle as O

    pool = lipz_synth.blob_pool(SEED, n=POOL_N, dim=X_DIM)
    arch = O.Arch(precision="bf16", batch=BATCH)
    # a state for the whole grid (initialisation is not part of the timed sample)
    state = _oracle_state(arch)
    nbr = O.neighbors(ROWS, COLS)
    done, t0 = 0, time.perf_counter()
    c = 0
    while True:
        cells = [c]
        data = O.batches(state, pool, cells=cells)
        prev = state if stale else None  # the same work; the sample's weights are synthetic
        ev = O.eval_neighborhoods(state, data, cells=cells, prev=prev)
        if mixture:
            O.mixture_update(state, data, cells=cells, prev=prev)
        a = state.arch
        sg = O.select_slot(ev["fG"][c], O.draw_words(state.seed, O.STREAM_TOUR_G, state.t, c,
                                                     a.tournament_size), a)
        sd = O.select_slot(ev["fD"][c], O.draw_words(state.seed, O.STREAM_TOUR_D, state.t, c,
                                                     a.tournament_size), a)
        x, z = data[c]
        gG, gD, _ = O.pair_gradients(state.Gw[nbr[c][sg]], state.Dw[nbr[c][sd]], x, z, a)
        Gn = O.adam_step(state.Gw[nbr[c][sg]], state.Gm[nbr[c][sg]], state.Gv[nbr[c][sg]], 0,
                         gG, a.lr, a)
        Dn = O.adam_step(state.Dw[nbr[c][sd]], state.Dm[nbr[c][sd]], state.Dv[nbr[c][sd]], 0,
                         gD, a.lr, a)
        for k in range(1, train_steps):
            x, z = O.draw_batch(state.seed, state.t, c, pool, a, k)
            gG, gD, _ = O.pair_gradients(Gn[0], Dn[0], x, z, a)
            Gn = O.adam_step(*Gn, gG, a.lr, a)
            Dn = O.adam_step(*Dn, gD, a.lr, a)
        done += 1
        c = (c + 1) % CELLS
        el = time.perf_counter() - t0
        if el >= seconds or (max_cells and done >= max_cells):
            return done, el


_STATE_CACHE = {}


def _oracle_state(arch):
    """Oracle grid state for the workload: Xavier weights from the seed (cells drawn lazily would
    change nothing: every cell's weights come from its own Philox stream)."""
    from oracle import lipz_oracle as O
    if "s" not in _STATE_CACHE:
        _STATE_CACHE["s"] = O.create(ROWS, COLS, arch, SEED)
    return _STATE_CACHE["s"]


def _threads():
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(k):
            return int(os.environ[k])
    return os.cpu_count() or 1


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo), and its logical core count."""
    name = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            k, _, v = line.partition(":")
            if k.strip() == "Model name" and v.strip():
                name = v.strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    if not name:
        try:
            with open("/proc/cpuinfo") as f:
                for line in f:
                    k, _, v = line.partition(":")
                    if k.strip() in ("model name", "Hardware", "CPU part") and v.strip():
                        name = v.strip()
                        break
        except OSError:
            pass
    return "%s, %d logical cores" % (name or "unknown CPU", os.cpu_count() or 0)


def _single_thread_sample(seconds):
    """The same oracle sample in a fresh interpreter with one BLAS / OpenMP thread (the thread
    count of a BLAS library is fixed when it loads)."""
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
    code = ("import json, bench; d, e = bench._oracle_sample(%r); print(json.dumps([d, e]))"
            % float(seconds))
    try:
        out = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True,
                             text=True, timeout=seconds * 4 + 120)
        done, el = json.loads(out.stdout.strip().splitlines()[-1])
    except (OSError, subprocess.SubprocessError, ValueError, IndexError):
        return None
    return {"value": 25.0 * done / el, "unit": UNIT, "cores": 1,
            "sample": "%d cells, %.1f s, one thread" % (done, el)}


def cpu_baseline(seconds, single_seconds=None):
    done, el = _oracle_sample(seconds)
    out = {"value": 25.0 * done / el, "unit": UNIT, "cores": _threads(), "kind": "oracle",
           "sample": "%d cells of the 12x12 bf16 B=100 workload (eval of 25 pairs + selection + "
                     "gradients + Adam per cell), %.1f s, numpy float64 + OpenBLAS" % (done, el),
           "cpu_model": cpu_model()}
    if single_seconds:
        out["single_thread"] = _single_thread_sample(single_seconds)
    return out


# ---- DCGAN workload (the 3x3 DCGAN configuration: width 64, z = 100, B = 128, bf16) --------
DC_ROWS, DC_COLS, DC_B, DC_Z, DC_W, DC_POOL = 3, 3, 128, 100, 64, 2000
DC_CELLS = DC_ROWS * DC_COLS
DC_PAIRS = 25 * DC_CELLS
DC_WORKLOAD = ("3x3 torus DCGAN G/D (512/256/128/64 channels, 64x64x3) bf16 B=128 "
               "(225 pairs/iter)")


def _dc_macs():
    """Algorithmic multiply-adds per sample: generator (transposed convolutions) and
    discriminator (convolutions), each layer H_in W_in C_in C_out 16 for the generator and
    H_out W_out C_in C_out 16 for the discriminator."""
    g, d, z = DC_W, DC_W, DC_Z
    gm = z * 8 * g * 16 + 16 * 8 * g * 4 * g * 16 + 64 * 4 * g * 2 * g * 16 \
        + 256 * 2 * g * g * 16 + 1024 * g * 3 * 16
    dm = 1024 * d * 3 * 16 + 256 * 2 * d * d * 16 + 64 * 4 * d * 2 * d * 16 \
        + 16 * 8 * d * 4 * d * 16 + 8 * d * 16
    return gm, dm


def run_dcgan(args):
    """The DCGAN grid iteration: device time per iteration, phases against the sustained bf16
    tensor rate (the convolutions of widths that fill the tiles run on tcgen05), end to end
    with host minibatches, and the oracle's rate."""
    import numpy as np
    import torch
    dist, rank, world = _dist()
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    import __graft_entry__
    __graft_entry__.build()
    import lipz_synth
    import paper_1811_12843_gb300 as L
    pool = lipz_synth.field_pool(SEED, n=DC_POOL)
    g = L.Grid(DC_ROWS, DC_COLS, seed=SEED + rank, precision="bf16", batch=DC_B, kind=1,
               x_dim=12288, z_dim=DC_Z, ngf=DC_W, ndf=DC_W, lr=5e-5,
               stale_neighbors=1 if args.stale_neighbors else 0,
               mixture=1 if args.mixture else 0)
    g.set_data(pool)
    stream = torch.cuda.Stream()
    g.set_stream(stream.cuda_stream)
    for _ in range(args.warmup):
        L.lipz_iterate(g.h, 1)
    g.synchronize()
    L.lipz_profile_read(g.h)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    with Clocks(local) as clk:
        e0.record(stream)
        for _ in range(args.steps):
            L.lipz_iterate(g.h, 1)
        e1.record(stream)
        g.synchronize()
    if dist:
        dist.barrier()
    ms = allreduce_max(dist, e0.elapsed_time(e1))
    launches = sum(v[2] for v in L.lipz_profile_read(g.h).values())
    ms_step = ms / args.steps
    value = DC_PAIRS * world * 1000.0 / ms_step
    L.lipz_profile_enable(g.h, True)
    for _ in range(max(2, args.steps // 2)):
        L.lipz_iterate(g.h, 1)
    prof = L.lipz_profile_read(g.h)
    L.lipz_profile_enable(g.h, False)
    phase_ms = {k: v[0] / max(v[1], 1) for k, v in prof.items()}
    # end to end: pinned host minibatches in, fitness out
    xs = [torch.from_numpy(pool[np.random.default_rng(i).integers(0, DC_POOL, DC_CELLS * DC_B)]
                           .reshape(DC_CELLS, DC_B, 12288)).pin_memory() for i in range(2)]
    fit = [(torch.zeros((DC_CELLS, 5), dtype=torch.float32).pin_memory(),
            torch.zeros((DC_CELLS, 5), dtype=torch.float32).pin_memory()) for _ in range(2)]
    L.lipz_iterate_batch(g.h, xs[0], fit[0][0], fit[0][1])
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    n_e2e = max(2, args.steps // 2)
    for i in range(n_e2e):
        L.lipz_iterate_batch_async(g.h, xs[i % 2], xs[(i + 1) % 2] if i + 1 < n_e2e else None,
                                   fit[i % 2][0], fit[i % 2][1])
    L.lipz_synchronize(g.h)
    e2e = DC_PAIRS * world * n_e2e / allreduce_max(dist, time.perf_counter() - t0)
    if rank != 0:
        return None
    hbm, tf_burst, tf_sus, kind = _peaks()
    gm, dm = _dc_macs()
    work = {"g_fwd": 2.0 * DC_CELLS * 5 * DC_B * gm, "d_fwd": 2.0 * DC_CELLS * 30 * DC_B * dm,
            "train_bwd": 2.0 * DC_CELLS * DC_B * (3 * gm + 7 * dm)}
    roofs = {}
    for ph, flop in work.items():
        t = phase_ms.get(ph)
        if t and t == t:
            ach = flop / (t * 1e-3) / 1e12
            roofs[ph] = {"bound": "tensor", "achieved": ach, "peak": tf_burst,
                         "unit": "TFLOP/s", "frac": ach / tf_burst, "traffic": None,
                         "algorithmic_flop": flop,
                         "peak_source": "%s burst bf16 (cuBLAS)" % kind}
    dom = max(roofs, key=lambda k: phase_ms[k])
    roof = dict(roofs[dom], phase=dom)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded smooth Gaussian random fields, 3x64x64, standing in for "
                "CelebA)",
        "config": {"workload": _workload(args), "rows": DC_ROWS, "cols": DC_COLS,
                   "global_batch": DC_B, "pairs_per_iter": DC_PAIRS,
                   "parallelism": "replicas" if world > 1 else "single",
                   "l2": "inputs larger than L2 (population and activations, several GB)"},
        "grid_iterations_per_sec": 1000.0 * world / ms_step,
        "phase_ms": phase_ms, "roofline": roof, "phase_rooflines": roofs,
        "e2e": {"value": e2e, "unit": UNIT, "h2d_bytes_per_step": DC_CELLS * DC_B * 12288 * 4,
                "d2h_bytes_per_step": 2 * DC_CELLS * 5 * 4 + 8 * 4},
        "gpu_launches": launches, "clocks": clk.summary(),
    }
    if world == 1 and not args.no_cpu_baseline:
        done, el = _dc_oracle_sample()
        line["cpu_baseline"] = {"value": 25.0 * done / el, "unit": UNIT, "cores": _threads(),
                                "kind": "oracle", "cpu_model": cpu_model(),
                                "sample": "%d cell(s) of the 3x3 DCGAN workload (evaluation of "
                                          "25 pairs), %.1f s" % (done, el)}
    return line


def _dc_oracle_sample(cells=1):
    import lipz_synth
    from oracle import lipz_oracle as O
    pool = lipz_synth.field_pool(SEED, n=DC_POOL)
    a = O.Arch(kind="dcgan", precision="bf16", batch=DC_B, z_dim=DC_Z, x_dim=12288, ngf=DC_W,
               ndf=DC_W)
    s = O.create(DC_ROWS, DC_COLS, a, SEED)
    t0 = time.perf_counter()
    for c in range(cells):
        O.eval_neighborhoods(s, O.batches(s, pool, cells=[c]), cells=[c])
    return cells, time.perf_counter() - t0


def _workload(args):
    if getattr(args, "dcgan", False):
        w = DC_WORKLOAD
        if args.stale_neighbors:
            w += ", stale neighbours"
        if args.mixture:
            w += ", mixture ES step"
        return w
    w = WORKLOAD
    if args.train_steps != 1:
        w += ", %d minibatch steps per iteration" % args.train_steps
    if args.mixture:
        w += ", mixture ES step"
    if args.stale_neighbors:
        w += ", stale neighbours"
    return w


def run_reference_dcgan(args):
    """The oracle on the DCGAN workload: each step evaluates one cell's 25 pairs."""
    _, rank, world = _dist()
    if rank != 0:
        return None
    total, el = 0, 0.0
    for _ in range(args.steps):
        d, e = _dc_oracle_sample()
        total += d
        el += e
    value = 25.0 * total / el
    return {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1000.0 * el / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded smooth Gaussian random fields, 3x64x64)",
            "config": {"workload": _workload(args), "rows": DC_ROWS, "cols": DC_COLS,
                       "global_batch": DC_B, "pairs_per_iter": DC_PAIRS, "parallelism": "cpu"},
            "impl": "reference",
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": _threads(), "kind": "oracle",
                             "sample": "1 cell per step of the 3x3 DCGAN workload",
                             "cpu_model": cpu_model()},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def run_reference(args):
    _, rank, world = _dist()
    if rank != 0:
        return None
    from oracle import lipz_oracle as O
    arch = O.Arch(precision="bf16", batch=BATCH)
    _oracle_state(arch)
    per_step_cells = 1
    for _ in range(args.warmup):
        _oracle_sample(1e9, max_cells=1, train_steps=args.train_steps, mixture=args.mixture,
                       stale=args.stale_neighbors)
    times = []
    total_cells = 0
    for _ in range(args.steps):
        done, el = _oracle_sample(1e9, max_cells=per_step_cells, train_steps=args.train_steps,
                                  mixture=args.mixture, stale=args.stale_neighbors)
        times.append(el)
        total_cells += done
    el = sum(times)
    value = 25.0 * total_cells / el
    return {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1000.0 * el / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded 10-blob 784-dim pool standing in for MNIST)",
            "config": {"workload": _workload(args), "rows": ROWS, "cols": COLS,
                       "global_batch": BATCH, "train_steps": args.train_steps,
                       "pairs_per_iter": PAIRS, "parallelism": "cpu"},
            "impl": "reference",
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": _threads(), "kind": "oracle",
                             "sample": "%d cells per step of the 12x12 bf16 B=100 workload"
                                       % per_step_cells, "cpu_model": cpu_model()},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=500)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--cpu-seconds-single", type=float, default=10.0,
                    help="seconds of the one-thread oracle sample (0: skip it)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end pass")
    ap.add_argument("--no-phases", action="store_true", help="skip the per-phase timing pass")
    ap.add_argument("--train-steps", type=int, default=1,
                    help="Adam steps per grid iteration (the later ones on fresh minibatches)")
    ap.add_argument("--mixture", action="store_true",
                    help="add the generator-mixture ES step to every iteration")
    ap.add_argument("--stale-neighbors", action="store_true",
                    help="neighbours seen one iteration late (asynchronous cells)")
    ap.add_argument("--dcgan", action="store_true",
                    help="the 3x3 DCGAN workload (tensor-core convolutions) instead of the MLP")
    ap.add_argument("--grid", default=None, metavar="RxC",
                    help="the MLP workload on a smaller or larger torus (for kernel captures on a "
                         "small case; not the benchmark configuration; no ncu traffic figures)")
    ap.add_argument("--dcgan-grid", default=None, metavar="RxC",
                    help="with --dcgan: a smaller or larger torus of the same networks (for "
                         "kernel captures on a small case; not the benchmark configuration)")
    args = ap.parse_args()
    if args.grid:
        global ROWS, COLS, WORKLOAD, PHASE_TRAFFIC
        ROWS, COLS = (int(v) for v in args.grid.lower().split("x"))
        _derive()
        WORKLOAD = "%dx%d torus MLP G/D bf16 B=100 (%d pairs/iter)" % (ROWS, COLS, PAIRS)
        PHASE_TRAFFIC = {}
    if args.dcgan_grid:
        global DC_ROWS, DC_COLS, DC_CELLS, DC_PAIRS, DC_WORKLOAD
        DC_ROWS, DC_COLS = (int(v) for v in args.dcgan_grid.lower().split("x"))
        DC_CELLS = DC_ROWS * DC_COLS
        DC_PAIRS = 25 * DC_CELLS
        DC_WORKLOAD = ("%dx%d torus DCGAN G/D (512/256/128/64 channels, 64x64x3) bf16 B=128 "
                       "(%d pairs/iter)" % (DC_ROWS, DC_COLS, DC_PAIRS))
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    if args.dcgan and args.impl == "reference":
        line = run_reference_dcgan(args)
    elif args.dcgan:
        line = run_dcgan(args)
    else:
        line = run_reference(args) if args.impl == "reference" else run_ours(args)
    if line is not None:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()

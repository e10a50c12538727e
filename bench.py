#!/usr/bin/env python
"""Throughput of the FPO pseudogradient update on GB300.

One step = fpo_error_signal (final RMSNorm forward, logits pass with the
log-sum-exp and the anchored probabilities, the row factors of E = s(softmax - onehot),
projection g = E W_U, final-norm VJP) + fpo_layer_update_grouped over every target
layer (G_l = g~^T A_l, W_master -= lr G_l, bf16 weights out), on the synthetic
OLMo-2-7B-shaped workload by default.  Prints one JSON line on rank 0.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl fpo|reference]

N > 1 runs N independent replicas (one per GPU, launched by torch.distributed.run):
the path has no exchange step between replicas, so there is no collective on the
data path; a barrier and a max over ranks bracket the timing.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "FPO update tokens/s and TFLOP/s at 1 GB300; fraction of dense BF16 roofline"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# --------------------------------------------------------------------------- helpers
def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def algorithmic_flops(wl):
    """4 T V d (logits once + projection) + 2 L T d d_ff."""
    return 4.0 * wl.T * wl.V * wl.d + 2.0 * wl.layers * wl.T * wl.d * wl.d_ff


def executed_flops(wl):
    """Adds the second logits GEMM of the two-pass (recompute) design: + 2 T V d."""
    return algorithmic_flops(wl) + 2.0 * wl.T * wl.V * wl.d


# Dense bf16 tcgen05 rate per SM and clock: 2 x 4096 multiply-adds (NVIDIA's nominal
# 2.25 PFLOP/s dense bf16 over 152 SMs at ~1.8 GHz).  The measured cuBLAS figures above
# reach ~94% of it per clock.
BF16_FLOP_PER_SM_CLOCK = 8192


def tensor_peak_at_clock(sm_count, sm_mhz):
    """Dense bf16 tensor-core peak (TFLOP/s) of the whole GPU at the sampled median clock."""
    if not sm_count or not sm_mhz:
        return None
    return BF16_FLOP_PER_SM_CLOCK * sm_count * sm_mhz * 1e6 / 1e12


def algorithmic_bytes(wl):
    esz = 2 if wl.dtype == "bf16" else 4
    return (wl.T * wl.d * esz + wl.V * wl.d * esz + wl.layers * wl.T * wl.d_ff * esz + wl.T * 4
            + wl.T * wl.d * esz + wl.layers * wl.d * wl.d_ff * (4 + 4 + esz))


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.dev), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons, power = [], None, set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
                power.append(float(parts[3]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": ["no samples"]}
        loaded = [s for s, p in zip(sm, power) if p > 0.5 * max(power)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm),
                "power_w_max": max(power) if power else None}


def max_over_ranks(x, device="cpu"):
    """Max of a per-rank scalar over all ranks (the slowest replica sets the time)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.item()


def whole_job_tokens_per_s(tokens_per_rank, world, max_ms):
    """Whole-job throughput: the tokens every replica processed over the slowest time."""
    return tokens_per_rank * world / (max_ms / 1e3)


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


# --------------------------------------------------------------------------- oracle baseline
_CPU_INPUTS = {}


def _cpu_inputs(wl):
    """The workload's inputs generated once on the host (seeded, as on the device)."""
    import synth
    if wl.name not in _CPU_INPUTS:
        _CPU_INPUTS[wl.name] = {
            "h": synth.make_h(wl), "w": synth.make_norm_w(wl), "W_U": synth.make_W_U(wl),
            "y": synth.make_targets(wl), "A0": synth.make_A(wl, 0),
            "W0": synth.make_W_master(wl, 0).numpy()}
    return _CPU_INPUTS[wl.name]


def oracle_sample(wl, n_tok, seed=0):
    """Time the fp64 CPU oracle on n_tok tokens of the workload and extrapolate to one
    step of T tokens: t_step = T * (per-token error signal + per-token G accumulation)
    + per-step weight update.  Inputs come from the same seeded generators."""
    import torch

    import oracle
    import synth

    oracle.build()
    inp = _cpu_inputs(wl)
    n_tok = min(n_tok, wl.T)
    gen = torch.Generator().manual_seed(1234 + seed)
    rows = torch.randperm(wl.T, generator=gen)[:n_tok].sort().values
    hn = synth.to_numpy_exact(inp["h"][rows])
    wn = synth.to_numpy_exact(inp["w"])
    Un = synth.to_numpy_exact(inp["W_U"])
    An = synth.to_numpy_exact(inp["A0"][rows])
    yn = inp["y"][rows].numpy()

    t0 = time.perf_counter()
    es = oracle.error_signal(hn, wn, Un, yn, eps=wl.eps, min_rms=wl.min_rms, s=1.0 / wl.T)
    t1 = time.perf_counter()
    G = oracle.pseudograd(es["g_tilde"], An)
    t2 = time.perf_counter()
    oracle.sgd_update(inp["W0"], G, wl.lr)
    t3 = time.perf_counter()
    per_tok = (t1 - t0) / n_tok + wl.layers * (t2 - t1) / n_tok
    step_s = wl.T * per_tok + wl.layers * (t3 - t2)
    return {"sample_s": t3 - t0, "step_s": step_s, "tokens_per_s": wl.T / step_s,
            "n_tok": n_tok, "es_s": t1 - t0, "G_s": t2 - t1, "upd_s": t3 - t2}


def copy_schedule(requested, copy_alone_ms, gemm_phase_ms):
    """The end-to-end input-copy schedule: `requested` unless it is "auto", which takes
    the per-phase parts ("sm") when one step's copy, timed alone, fits in the error
    signal's GEMM phases, else one copy launch per step ("sm1")."""
    if requested != "auto":
        return requested
    return "sm" if copy_alone_ms <= gemm_phase_ms else "sm1"


def cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def cpu_model():
    """The host CPU's model name (lscpu), for the CPU-baseline record."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    import platform
    return platform.processor() or platform.machine()


def sample_text(r, wl):
    return (f"{r['n_tok']} of {wl.T} tokens through the oracle (error signal {r['es_s']:.2f} s, "
            f"G for 1 of {wl.layers} layers {r['G_s']:.2f} s, one weight update {r['upd_s']:.2f} s),"
            f" extrapolated to one {wl.T}-token step of {wl.layers} layers: "
            f"T*(t_es+L*t_G)/n + L*t_upd")


def run_reference(args, wl):
    world, rank, _ = dist_setup()
    if rank != 0:
        return
    # the oracle runs one token per thread at a time, so a sample is a whole number of
    # tokens per host thread (1 to 4, fewer for longer runs) to keep every core busy
    n_tok = args.ref_tokens or cores() * max(1, min(4, 40 // max(1, args.warmup + args.steps)))
    steps = []
    for i in range(args.warmup + args.steps):
        r = oracle_sample(wl, n_tok, seed=i)
        if i >= args.warmup:
            steps.append(r)
    step_s = statistics.median(r["step_s"] for r in steps)
    sample_s = statistics.median(r["sample_s"] for r in steps)
    value = wl.T / step_s
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        # not timed whole: a T-token step of the oracle takes minutes to hours, so each step
        # times a bounded sample and this is that sample extrapolated to one T-token step
        "ms_per_step": step_s * 1e3, "ms_per_step_kind": "extrapolated",
        "timing": (f"extrapolated: each of the {args.steps} timed steps runs {n_tok} of "
                   f"{wl.T} tokens (median wall time {sample_s * 1e3:.0f} ms per sampled "
                   f"step) and scales the per-token cost to the whole step"),
        "sample_ms_per_step": sample_s * 1e3,
        "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(wl, args),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores(),
                         "cpu_model": cpu_model(), "kind": "oracle",
                         "sample": sample_text(steps[-1], wl)},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def workload_config(wl, args):
    return {"workload": wl.name, "T": wl.T, "d": wl.d, "d_ff": wl.d_ff, "V": wl.V,
            "target_layers": wl.layers, "targets": "zipf(1.1)" if wl.targets == "zipf" else wl.targets,
            "lr": wl.lr, "t_chunk": min(args.t_chunk or AUTO_T_CHUNK, wl.T),
            "global_batch_tokens": wl.T * args.gpus,
            "error_matrix": {"auto": "direct (auto)", "recompute": "recompute",
                             "stored": "stored-logits", "direct": "direct"}[args.algo],
            "norms_composed": "final" + (" + post-FFN per layer" if args.post_ffn_norm else "")
                              + (" + pre-MLP per layer" if args.pre_mlp_norm else ""),
            "weights_updated": ("W3, W1, W2 (W1/W2 via W3_init feedback, the same optimizer)"
                                if args.gate_up else "W3"),
            "optimizer": ("plain SGD fused in the update GEMM epilogue" if args.optimizer == "fused-sgd"
                          else f"{args.optimizer} on fp32 masters, clip={args.clip} (1% of ||W||_F)"),
            "l2": "inputs larger than L2 (W_U %.0f MB, A_l %.2f GB per step); no flush"
                  % (wl.V * wl.d * 2 / 1e6, wl.layers * wl.T * wl.d_ff * 2 / 1e9),
            **({"inputs": "window stress: +-1 hidden states, W_U x 64"}
               if getattr(args, "window_stress", False) else {})}


# --------------------------------------------------------------------------- GPU arm
def run_fpo(args, wl):
    import torch
    import torch.distributed as dist

    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    import paper_2608_14563_gb300 as fpo
    import synth

    if args.gemm_variant >= 0:
        fpo.set_gemm_variant(args.gemm_variant)
    variant = fpo.set_gemm_variant(-1)  # read back (a negative value changes nothing)
    if args.band:
        fpo._lib.fpo_testing_set_band(args.band)

    wl_r = synth.Workload(wl.name, T=wl.T, d=wl.d, d_ff=wl.d_ff, V=wl.V, layers=wl.layers,
                          dtype=wl.dtype, targets=wl.targets, lr=wl.lr, seed=rank)
    dev = torch.device("cuda", local)
    h = synth.make_h(wl_r, dev)
    w = synth.make_norm_w(wl_r, dev)
    W_U = synth.make_W_U(wl_r, dev)
    y = synth.make_targets(wl_r, dev)
    if args.window_stress:
        # logits ~30x the usual scale (+-1 hidden states, W_U x 64): most tokens fall
        # outside the direct algorithm's anchor window and are recomputed by its fixup
        h = torch.where(h >= 0, 1.0, -1.0).to(h.dtype)
        W_U = (W_U.float() * 64).to(W_U.dtype)
    A = [synth.make_A(wl_r, l, dev) for l in range(wl.layers)]
    Wm = [synth.make_W_master(wl_r, l, dev) for l in range(wl.layers)]
    Wo = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev) for _ in range(wl.layers)]
    g = torch.empty_like(h)
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    post = args.post_ffn_norm
    pre = args.pre_mlp_norm
    layer_norms = post or pre  # per-layer signals g~^(l) (Sec. 3.2)
    gate_up = args.gate_up
    if gate_up:  # SwiGLU caches, W3_init feedback, gate/up masters and signal buffers
        gu_ab = [synth.make_gate_up(wl_r, l, dev) for l in range(wl.layers)]
        gu_x = [synth.make_mlp_in(wl_r, l, dev) for l in range(wl.layers)]
        gu_W3 = [synth.make_W_master(wl_r, l, dev).to(torch.bfloat16) for l in range(wl.layers)]
        gu_W12 = [m for l in range(wl.layers) for m in synth.make_gate_up_master(wl_r, l, dev)]
        gu_out = [torch.empty(wl.d_ff, wl.d, dtype=torch.bfloat16, device=dev) for _ in gu_W12]
        gu_sig = [torch.empty(wl.T, wl.d_ff, dtype=torch.bfloat16, device=dev)
                  for _ in range(2 * wl.layers)]
        ws_gu = torch.empty(fpo.layer_update_workspace(), dtype=torch.uint8, device=dev)
    if post:  # per-layer MLP outputs and post-FFN norm weights
        m_out = [synth.make_mlp_out(wl_r, l, dev) for l in range(wl.layers)]
        gp = [synth.make_post_norm_w(wl_r, l, dev) for l in range(wl.layers)]
    if pre:  # per-layer pre-MLP norm inputs (residual stream) and weights
        x_pre = [synth.make_pre_norm_in(wl_r, l, dev) for l in range(wl.layers)]
        gq = [synth.make_pre_norm_w(wl_r, l, dev) for l in range(wl.layers)]
    if layer_norms:  # the layer-specific signals
        g_l = [torch.empty_like(h) for _ in range(wl.layers)]
    algo = {"auto": fpo.ES_AUTO, "recompute": fpo.ES_RECOMPUTE,
            "stored": fpo.ES_STORED_LOGITS, "direct": fpo.ES_DIRECT}[args.algo]
    # the algorithm that runs (bf16: AUTO is the direct algorithm)
    algo_name = {fpo.ES_RECOMPUTE: "recompute", fpo.ES_STORED_LOGITS: "stored-logits"}.get(
        algo, "direct")
    desc = fpo.error_signal_desc(wl.T, wl.d, wl.V, fpo.BF16, eps=wl.eps, min_rms=wl.min_rms,
                                 t_chunk=args.t_chunk, algo=algo)
    ws_es = torch.empty(fpo.error_signal_workspace(desc), dtype=torch.uint8, device=dev)
    ws_up = torch.empty(fpo.layer_update_workspace(), dtype=torch.uint8, device=dev)
    optimize = args.optimizer != "fused-sgd"
    if optimize:
        kind = {"sgd": fpo.OPT_SGD, "sgdm": fpo.OPT_SGD_MOMENTUM, "adamw": fpo.OPT_ADAMW}[
            args.optimizer]
        clip = {"none": fpo.CLIP_NONE, "step": fpo.CLIP_STEP, "grad": fpo.CLIP_GRADIENT}[args.clip]
        opt = fpo.optimizer_desc(kind, lr=wl.lr, clip=clip, step=10)
        st1 = ([torch.zeros(wl.d, wl.d_ff, device=dev) for _ in range(wl.layers)]
               if kind != fpo.OPT_SGD else None)
        st2 = ([torch.zeros(wl.d, wl.d_ff, device=dev) for _ in range(wl.layers)]
               if kind == fpo.OPT_ADAMW else None)
        ws_up = torch.empty(fpo.layer_optimize_workspace(wl.layers, wl.d, wl.d_ff),
                            dtype=torch.uint8, device=dev)
        if gate_up:  # the same optimizer and clip on W1 and W2 of every target layer
            gu_st1 = ([torch.zeros(wl.d_ff, wl.d, device=dev) for _ in range(2 * wl.layers)]
                      if kind != fpo.OPT_SGD else None)
            gu_st2 = ([torch.zeros(wl.d_ff, wl.d, device=dev) for _ in range(2 * wl.layers)]
                      if kind == fpo.OPT_ADAMW else None)
            ws_gu_opt = torch.empty(fpo.layer_optimize_workspace(2 * wl.layers, wl.d_ff, wl.d),
                                    dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    # The tensors one step reads that come from the forward pass / the data: the
    # end-to-end loop below copies them from host memory every step.
    X0 = {"h": h, "y": y, "A": A, "m": m_out if post else [], "xpre": x_pre if pre else [],
          "ab": [t for pair in gu_ab for t in pair] if gate_up else [],
          "x": gu_x if gate_up else []}

    ratio = args.norm_ratio
    # Sec. 2.2 diagnostic: cos(G_l, G~_l) per target layer against a 'true' gradient G~_l
    # (a seeded stand-in drawn once: the timing does not depend on its values), on by
    # default for the diag workload
    cosine = args.cosine or wl.name.startswith("diag")
    if (ratio or cosine) and optimize:
        raise SystemExit("--norm-ratio / --cosine read G_l from the fused update "
                         "(--optimizer fused-sgd)")
    if ratio or cosine:
        Go = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev)
              for _ in range(wl.layers)]
    if ratio:  # App. C update-magnitude ratio on each step's G_l (bf16) and fp32 masters
        ratio_out = torch.empty(wl.layers, 4, dtype=torch.float64, device=dev)
        ws_nr = torch.empty(fpo.norm_ratio_workspace(wl.layers, wl.d * wl.d_ff),
                            dtype=torch.uint8, device=dev)
    if cosine:
        n_el = wl.d * wl.d_ff
        G_true = [synth.make_noise(n_el, seed=wl_r.seed, layer=l, device=dev).mul_(1e-3)
                  .to(torch.bfloat16) for l in range(wl.layers)]
        cos_out = torch.empty(wl.layers, 4, dtype=torch.float64, device=dev)
        ws_cos = torch.empty(fpo.cosine_grouped_workspace(wl.layers, n_el), dtype=torch.uint8,
                             device=dev)
        Go_flat = [x.view(-1) for x in Go]
    # the diagnostic's step (G_l only, no master to move) forms the cosines in the update
    # GEMM's epilogue, so G_l is not read back, unless asked to run the two calls
    fused_cos = (cosine and wl.lr == 0.0 and not (layer_norms or optimize or ratio or gate_up)
                 and not args.cosine_separate)
    if fused_cos:
        G_true_2d = [x.view(wl.d, wl.d_ff) for x in G_true]
        ws_gc = torch.empty(fpo.layer_grad_cosine_workspace(wl.layers, wl.d, wl.d_ff),
                            dtype=torch.uint8, device=dev)

    def update(X):
        signals = g_l if layer_norms else [g] * wl.layers
        G_outs = Go if (ratio or cosine) else None
        if optimize:
            fpo.layer_optimize_grouped(signals, X["A"], opt, Wm, W_outs=Wo, states1=st1,
                                       states2=st2, workspace=ws_up)
        elif layer_norms:
            fpo.layer_update_grouped_signals(g_l, X["A"], wl.lr, W_masters=Wm, W_outs=Wo,
                                             G_outs=G_outs, workspace=ws_up)
        elif fused_cos:
            # the diagnostic's step: G_l and its cosine against the true gradient
            fpo.layer_grad_cosine_grouped(g, X["A"], G_true_2d, Go, out=cos_out, workspace=ws_gc)
        elif wl.lr == 0.0 and G_outs is not None:
            # the diagnostic's step: G_l only (no master to move at lr = 0)
            fpo.layer_update_grouped(g, X["A"], 0.0, G_outs=G_outs, workspace=ws_up)
        else:
            fpo.layer_update_grouped(g, X["A"], wl.lr, W_masters=Wm, W_outs=Wo, G_outs=G_outs,
                                     workspace=ws_up)

    def gate_up_update(X):
        for l in range(wl.layers):
            fpo.gate_up_signals(g_l[l] if layer_norms else g, gu_W3[l], X["ab"][2 * l],
                                X["ab"][2 * l + 1], gu_sig[2 * l], gu_sig[2 * l + 1],
                                workspace=ws_gu)
        gu_act = [x for x in X["x"] for _ in range(2)]
        if optimize:
            fpo.layer_optimize_grouped(gu_sig, gu_act, opt, gu_W12, W_outs=gu_out,
                                       states1=gu_st1, states2=gu_st2, workspace=ws_gu_opt)
        else:
            fpo.layer_update_grouped_signals(gu_sig, gu_act, wl.lr, W_masters=gu_W12,
                                             W_outs=gu_out, workspace=ws_gu)

    def step(X, stage_events=None, upd_events=None, per_chunk=False):
        fpo.error_signal(X["h"], w, W_U, X["y"], g, eps=wl.eps, min_rms=wl.min_rms,
                         t_chunk=args.t_chunk, loss_out=loss, workspace=ws_es,
                         stage_events=stage_events, algo=algo, per_chunk_events=per_chunk)
        if layer_norms:
            if upd_events:
                upd_events[2].record(stream)
            fpo.layer_signals(g, g_l, m=X["m"] if post else None, gamma_post=gp if post else None,
                              x=X["xpre"] if pre else None, gamma_pre=gq if pre else None,
                              eps=wl.eps, min_rms=wl.min_rms)
        if upd_events:
            upd_events[0].record(stream)
        update(X)
        if upd_events:
            upd_events[1].record(stream)
        if gate_up:
            gate_up_update(X)
            if upd_events:
                upd_events[3].record(stream)
        if ratio:
            if upd_events:
                upd_events[4].record(stream)
            fpo.norm_ratio(Go, Wm, rel_step=0.01, out=ratio_out, workspace=ws_nr)
            if upd_events:
                upd_events[5].record(stream)
        if cosine:
            if upd_events:
                upd_events[6].record(stream)
            if not fused_cos:  # (fused: already formed by the update's epilogue)
                fpo.cosine_grouped(Go_flat, G_true, out=cos_out, workspace=ws_cos)
            if upd_events:
                upd_events[7].record(stream)

    for _ in range(args.warmup):
        step(X0)
    torch.cuda.synchronize()
    ws_up_status = ws_gc if fused_cos else ws_up  # the update call's own status word
    assert (fpo.get_device_status(ws_es) == fpo.OK
            and fpo.get_device_status(ws_up_status) == fpo.OK)

    # per-stage events of every token chunk, for every timed step (recorded once so their
    # handles exist): 0 start, 1 after the RMSNorm forward, per chunk c the ends of its
    # logits pass (2+4c), combine (3+4c), fixup / E stage (4+4c) and projection (5+4c), and
    # the end of the VJP (2+4n)
    n_ev = fpo.stage_event_count(fpo.error_signal_desc(
        wl.T, wl.d, wl.V, fpo.BF16, t_chunk=args.t_chunk, algo=algo, per_chunk_events=True))
    n_chunks = (n_ev - 3) // 4
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(n_ev)] for _ in range(args.steps)]
    uev = [[torch.cuda.Event(enable_timing=True) for _ in range(8)] for _ in range(args.steps)]
    for e in [x for row in ev + uev for x in row]:
        e.record(stream)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    launches0 = fpo.kernel_launches()  # the library counts every kernel it launches
    start.record(stream)
    for i in range(args.steps):
        step(X0, ev[i], uev[i], per_chunk=True)
    end.record(stream)
    launches = fpo.kernel_launches() - launches0
    torch.cuda.synchronize()
    clk = clocks.stop()
    if world > 1:
        dist.barrier()
    ms = start.elapsed_time(end) / args.steps
    status = (fpo.get_device_status(ws_es), fpo.get_device_status(ws_up_status))
    # rows of the last step's last token chunk that the direct algorithm recomputed
    # outside its anchor window
    fixup_rows = (fpo.direct_fixup_rows(X0["h"], W_U, ws_es, t_chunk=args.t_chunk, algo=algo)
                  if algo_name == "direct" else None)

    # the direct algorithm's projection epilogue applies the final-norm VJP itself: its
    # "projection" stage includes the VJP and its "rmsnorm_vjp" stage is empty
    names = ["rmsnorm_fwd", "logits_lse_pass", "lse_combine",
             {"direct": "direct_fixup", "stored-logits": "logits_to_error",
              "recompute": "recompute_error_pass"}[algo_name], "projection", "rmsnorm_vjp"]
    def stage_sum(e, k):  # one kernel stage summed over the token chunks (k: 1..4)
        if k == 0:
            return e[0].elapsed_time(e[1])
        if k == 5:
            return e[5 + 4 * (n_chunks - 1)].elapsed_time(e[2 + 4 * n_chunks])
        total = 0.0
        for c in range(n_chunks):
            a = (1 if c == 0 else 5 + 4 * (c - 1)) if k == 1 else k + 4 * c
            total += e[a].elapsed_time(e[k + 1 + 4 * c])
        return total

    stage_ms = {n: statistics.mean(stage_sum(ev[i], k) for i in range(args.steps))
                for k, n in enumerate(names)}
    stage_ms["layer_update"] = statistics.mean(uev[i][0].elapsed_time(uev[i][1])
                                               for i in range(args.steps))
    if layer_norms:
        stage_ms["layer_signals"] = statistics.mean(uev[i][2].elapsed_time(uev[i][0])
                                                    for i in range(args.steps))
    if gate_up:
        stage_ms["gate_up"] = statistics.mean(uev[i][1].elapsed_time(uev[i][3])
                                              for i in range(args.steps))
    if ratio:
        stage_ms["norm_ratio"] = statistics.mean(uev[i][4].elapsed_time(uev[i][5])
                                                 for i in range(args.steps))
    if cosine:
        stage_ms["cosine"] = statistics.mean(uev[i][6].elapsed_time(uev[i][7])
                                             for i in range(args.steps))

    # ------------------------------------------------ end to end through the public API
    # Every step copies its inputs (h, targets, every A_l, and the per-layer caches of the
    # optional rows) from pinned host memory and reads the loss back.  The inputs rotate
    # through `depth` device sets: while step i computes on one set, the inputs of step
    # i + depth - 1 are copied into the set step i - 1 has finished reading, on a copy
    # stream, so copies may run up to depth - 1 steps ahead (slack for a host link whose
    # throughput stalls now and then).  Inside the timed region each step issues exactly
    # one step's copies, and the region ends only after the copy stream has drained.
    e2e = None
    if not args.no_e2e:
        def clone_set(X):
            return {k: (v.clone() if torch.is_tensor(v) else [t.clone() for t in v])
                    for k, v in X.items()}

        def flat(X):
            return [X["h"], X["y"]] + [t for k in ("A", "m", "xpre", "ab", "x") for t in X[k]]

        depth = max(2, args.e2e_depth)
        sets = [X0] + [clone_set(X0) for _ in range(depth - 1)]
        host = [t.cpu().pin_memory() for t in flat(X0)]
        loss_host = torch.empty(1, dtype=torch.float32).pin_memory()
        copy_stream = torch.cuda.Stream(device=dev)
        ready = [torch.cuda.Event() for _ in range(depth)]
        freed = [torch.cuda.Event() for _ in range(depth)]
        for e in freed:
            e.record(stream)

        # "sm": the copy of a step's inputs in one part per long GEMM phase of the error
        # signal (each token chunk's logits pass and projection), parts split by bytes,
        # each started at the stage boundary where its phase begins, so that the copies
        # run beside long GEMMs and not beside the short bandwidth-bound kernels between
        # them, which the copy's host loads slow down most
        sev = [torch.cuda.Event() for _ in range(n_ev)]
        for e in sev:
            e.record(stream)
        starts = [1 if c == 0 else 5 + 4 * (c - 1) for c in range(n_chunks)]  # logits begin
        triggers = sorted(starts + [4 + 4 * c for c in range(n_chunks)])        # + projections
        nbytes = [t.numel() * t.element_size() for t in host]
        cuts, acc, total = [0], 0, sum(nbytes)
        for j, nb in enumerate(nbytes):
            acc += nb
            if len(cuts) < len(triggers) and acc >= total * len(cuts) / len(triggers):
                cuts.append(j + 1)
        cuts.append(len(host))
        parts = [(a, b) for a, b in zip(cuts[:-1], cuts[1:]) if b > a]

        # one step's copy timed alone (the host link's own rate) decides the schedule: the
        # per-phase parts pay off while the copy fits beside the error signal's GEMM phases
        # (OLMo shape: e2e - device step 0.59 against 0.87 ms for one launch per step); a
        # copy longer than those phases spills beside the update either way, and there
        # one launch per step did better (Falcon shape: 3.7 against 6.4 ms)
        link_ms = float("inf")
        for _ in range(2):  # the first pass also maps the host pages
            t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            t0.record(copy_stream)
            fpo.h2d_copy(flat(sets[1]), host, stream=copy_stream)
            t1.record(copy_stream)
            torch.cuda.synchronize()
            link_ms = min(link_ms, t0.elapsed_time(t1))
        gemm_phase_ms = stage_ms["logits_lse_pass"] + stage_ms["projection"]
        copy_mode = copy_schedule(args.e2e_copy, link_ms, gemm_phase_ms)

        def prefetch(b, after=None):
            copy_stream.wait_event(freed[b])
            with torch.cuda.stream(copy_stream):
                dst = flat(sets[b])
                if copy_mode == "sm" and after is not None:
                    for (p0, p1), k in zip(parts, triggers):
                        copy_stream.wait_event(after[k])  # this part's GEMM phase begins
                        fpo.h2d_copy(dst[p0:p1], host[p0:p1], stream=copy_stream)
                elif copy_mode in ("sm", "sm1"):
                    fpo.h2d_copy(dst, host, stream=copy_stream)
                else:
                    for d_t, h_t in zip(dst, host):
                        d_t.copy_(h_t, non_blocking=True)
                ready[b].record(copy_stream)

        def e2e_step(i):
            b = i % depth
            stream.wait_event(ready[b])
            step(sets[b], sev, per_chunk=True)
            prefetch((i + depth - 1) % depth, sev)  # the inputs of step i + depth - 1
            freed[b].record(stream)
            loss_host.copy_(loss, non_blocking=True)

        for b in range(depth - 1):
            prefetch(b)
        for i in range(max(1, args.warmup)):
            e2e_step(i)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        s2, e2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s2.record(stream)
        e2e_l0 = fpo.kernel_launches()
        for i in range(max(1, args.warmup), max(1, args.warmup) + args.steps):
            e2e_step(i)
        e2e_launches = fpo.kernel_launches() - e2e_l0
        stream.wait_stream(copy_stream)
        e2.record(stream)
        torch.cuda.synchronize()
        e2e_ms = max_over_ranks(s2.elapsed_time(e2) / args.steps, dev)
        h2d = sum(t.numel() * t.element_size() for t in host)
        e2e = {"value": whole_job_tokens_per_s(wl.T, world, e2e_ms), "unit": "tokens/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": 4, "ms_per_step": e2e_ms,
               "gpu_launches": e2e_launches,
               "copy": {"sm": "fpo_h2d_copy (SM loads of mapped pinned memory): one launch per "
                              "long GEMM phase of the error signal (each token chunk's logits "
                              "pass and projection), started when the phase begins",
                        "sm1": "fpo_h2d_copy (SM loads of mapped pinned memory): one launch per "
                               "step",
                        "ce": "copy engines: one cudaMemcpyAsync per tensor"}[copy_mode],
               "copy_alone_ms": link_ms, "error_signal_gemm_ms": gemm_phase_ms,
               "pipeline": f"all step inputs H2D from pinned memory each step, {depth} device "
                           "sets: copies run on a copy stream up to "
                           f"{depth - 1} steps ahead of compute; loss D2H"}

    ms = max_over_ranks(ms, dev)

    if rank == 0:
        peaks, peaks_src = load_peaks()
        tok_s = whole_job_tokens_per_s(wl.T, world, ms)
        # the W1/W2 path adds error_h = g W3_init and the two gradient GEMMs per layer
        gu_flops = 6.0 * wl.layers * wl.T * wl.d * wl.d_ff if gate_up else 0.0
        alg_tf = (algorithmic_flops(wl) + gu_flops) / (ms / 1e3) / 1e12
        exe_tf = ((executed_flops(wl) if algo_name == "recompute" else algorithmic_flops(wl))
                  + gu_flops) / (
            ms / 1e3) / 1e12
        per_kernel_flops = {
            "logits_lse_pass": 2.0 * wl.T * wl.V * wl.d,
            "projection": 2.0 * wl.T * wl.V * wl.d,
            "layer_update": 2.0 * wl.layers * wl.T * wl.d * wl.d_ff,
        }
        if algo_name == "recompute":
            per_kernel_flops["recompute_error_pass"] = 2.0 * wl.T * wl.V * wl.d
        if gate_up:
            per_kernel_flops["gate_up"] = gu_flops
        # dominant kernel among those whose work is algorithmic (the recompute is overhead)
        dom = max(("logits_lse_pass", "projection", "layer_update"), key=lambda k: stage_ms[k])
        peak_sus = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
        achieved = per_kernel_flops[dom] / (stage_ms[dom] / 1e3) / 1e12
        roofline = {"bound": "tensor", "achieved": achieved, "peak": peak_sus, "unit": "TFLOP/s",
                    "frac": achieved / peak_sus,
                    "traffic": load_traffic(dom, {"workload": wl.name, "algo": algo_name,
                                                  "gemm_variant": variant,
                                                  "t_chunk": min(args.t_chunk or AUTO_T_CHUNK,
                                                                 wl.T),
                                                  "window_stress": bool(args.window_stress)}),
                    "kernel": dom, "peak_kind": f"bf16 sustained ({peaks_src})"}
        # the same kernel against the hardware's own dense bf16 rate at the clock it ran at
        # (the cuBLAS-based peaks above are themselves ~94% of it per clock)
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        tp = tensor_peak_at_clock(sms, clk.get("sm_mhz"))
        roofline["tensor_peak_at_clock"] = None if tp is None else {
            "tflops": tp, "frac": achieved / tp, "step_frac": alg_tf / tp,
            "basis": f"{BF16_FLOP_PER_SM_CLOCK} FLOP/SM/clock x {sms} SMs x median SM clock "
                     f"{clk.get('sm_mhz')} MHz under load"}
        cpu = None
        if world == 1 and not args.no_cpu:
            r = oracle_sample(wl, args.cpu_tokens)
            cpu = {"value": r["tokens_per_s"], "unit": "tokens/s", "cores": cores(),
                   "cpu_model": cpu_model(),
                   "kind": "oracle", "sample": sample_text(r, wl)}
        line = {
            "metric": METRIC, "value": tok_s, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": f"synthetic (seeded; {wl.name} workload: random weights and activations)",
            "config": workload_config(wl, args),
            "tflops": {"algorithmic": alg_tf, "executed": exe_tf,
                       "frac_of_bf16_peak_burst": alg_tf / peaks.get("bf16_tflops", 1900.0),
                       "frac_of_bf16_peak_sustained": alg_tf / peak_sus,
                       "peaks": peaks_src},
            "roofline": roofline,
            "kernels_ms": stage_ms,
            "kernels_note": ("the projection's epilogue applies the final-norm VJP (direct "
                             "algorithm): rmsnorm_vjp is an empty stage"
                             if algo_name == "direct" else None),
            "kernels_tflops": {k: per_kernel_flops[k] / (stage_ms[k] / 1e3) / 1e12
                               for k in per_kernel_flops},
            "kernels_gbs": {**({"norm_ratio": wl.layers * wl.d * wl.d_ff * (2 + 4)
                                / (stage_ms["norm_ratio"] / 1e3) / 1e9} if ratio else {}),
                            **({"cosine": wl.layers * wl.d * wl.d_ff * (2 + 2)
                                / (stage_ms["cosine"] / 1e3) / 1e9}
                               if cosine and not fused_cos else {}),
                            # per layer: g, the norm inputs and the signal, bf16 rows
                            **({"layer_signals": wl.layers * wl.T * wl.d * 2 * (2 + post + pre)
                                / (stage_ms["layer_signals"] / 1e3) / 1e9}
                               if layer_norms else {})},
            "cosine": cos_out[:, 3].tolist() if cosine else None,
            "cosine_mode": (None if not cosine else
                            "fused: fpo_layer_grad_cosine_grouped forms the sums in the update "
                            "GEMM's epilogue (the cosine stage is empty)" if fused_cos else
                            "separate: fpo_cosine_grouped reads G_l and G~_l after the update"),
            "norm_ratio": ({"ratio": ratio_out[:, 2].tolist(),
                            "implied_sgd_lr_1pct": ratio_out[:, 3].tolist()} if ratio else None),
            "algo": algo_name,
            "direct_fixup_rows_last_chunk": fixup_rows,
            "gemm_kernel": {0: "single-cta 128x256 (tcgen05 cta_group::1)",
                            1: "cta-pair 256x256 (tcgen05 cta_group::2; three 64 KB stages of "
                               "two k-blocks)",
                            2: "cta-pair 256x256 (three 64 KB stages of two k-blocks), projection "
                               "256x512 (tcgen05 cta_group::2)",
                            }[variant],
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": launches,
            "clocks": clk,
            "device_status": list(status),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# The library's token chunk when --t-chunk is 0 (FPO_AUTO_T_CHUNK in include/fpo.h).
AUTO_T_CHUNK = 8192

# Files that define each kernel whose DRAM traffic profiles/traffic.json records.
GEMM_SOURCES = ("tc_gemm.cuh", "tc_gemm_pair.cuh", "epilogues.cuh", "error_math.cuh", "ptx.cuh",
                "gemm_bf16.cu")
KERNEL_SOURCES = {
    "logits_lse_pass": GEMM_SOURCES,
    "projection": GEMM_SOURCES,
    "layer_update": GEMM_SOURCES,
    "logits_to_error": ("rowwise.cu", "error_math.cuh"),
}


def load_traffic(kernel, run_config):
    """Per-launch DRAM bytes of `kernel` from the committed ncu summary, or None when that
    summary is missing, was taken on another configuration (workload, algorithm, kernel
    variant, token chunk, inputs) or on different sources of that kernel."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path) or kernel not in KERNEL_SOURCES:
        return None
    with open(path) as f:
        tr = json.load(f)
    if tr.get("_config") != run_config:
        return None
    ent = tr.get(kernel)
    if not ent or ent.get("sources_sha256") != sources_digest(KERNEL_SOURCES[kernel]):
        return None
    return ent.get("bytes_per_launch")


def sources_digest(files):
    import hashlib
    csrc = os.path.join(ROOT, "paper_2608_14563_gb300", "csrc")
    hsh = hashlib.sha256()
    for name in sorted(files):
        with open(os.path.join(csrc, name), "rb") as f:
            hsh.update(name.encode() + f.read())
    return hsh.hexdigest()


def ensure_built():
    """Compile libfpo.so in-tree when it is missing (the package refuses to load without it)."""
    import importlib.util
    spec = importlib.util.spec_from_file_location(
        "_fpo_build", os.path.join(ROOT, "paper_2608_14563_gb300", "build.py"))
    b = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(b)
    b.build()


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    # Defaults measure the steady state: under sustained load the GPU's power limiter
    # settles after ~1 s (runs of 20 steps finish 4-5% faster), and the sustained bf16
    # peak the roofline uses was measured over 4 s of back-to-back GEMMs.
    ap.add_argument("--steps", type=int, default=200,
                    help="timed steps (~5 s at the OLMo shape: the power-capped steady state)")
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=("fpo", "reference"), default="fpo")
    ap.add_argument("--workload", default="olmo", help="olmo | qwen | falcon | diag")
    ap.add_argument("--t-chunk", type=int, default=0, help="tokens per E chunk (0 = all)")
    ap.add_argument("--optimizer", choices=("fused-sgd", "sgd", "sgdm", "adamw"),
                    default="fused-sgd",
                    help="fused-sgd: W -= lr G in the GEMM epilogue; otherwise G, the relative "
                         "clip and the optimizer step on the fp32 masters (fpo_layer_optimize_grouped)")
    ap.add_argument("--clip", choices=("none", "step", "grad"), default="step",
                    help="relative clip to 1%% of ||W||_F for --optimizer sgd/sgdm/adamw")
    ap.add_argument("--gate-up", action="store_true",
                    help="also update W1/W2 of every layer through the cached W3_init feedback")
    ap.add_argument("--post-ffn-norm", action="store_true",
                    help="compose each layer's post-FFN RMSNorm VJP (OLMo-2 layout) in the step")
    ap.add_argument("--pre-mlp-norm", action="store_true",
                    help="compose each layer's pre-MLP RMSNorm VJP (Qwen3 layout; with "
                         "--post-ffn-norm the Gemma 3 layout) in the step")
    ap.add_argument("--algo", choices=("auto", "recompute", "stored", "direct"), default="auto",
                    help="how the error matrix is formed (fpo_es_algo)")
    ap.add_argument("--cosine", action="store_true",
                    help="add the Sec. 2.2 diagnostic cosine of every layer's G_l to each step "
                         "(always on for the diag workload)")
    ap.add_argument("--cosine-separate", action="store_true",
                    help="diag workload: G_l by the grouped update, then fpo_cosine_grouped "
                         "(two calls) instead of fpo_layer_grad_cosine_grouped")
    ap.add_argument("--norm-ratio", action="store_true",
                    help="add the App. C update-magnitude ratio ||G_l||/||W_l|| to every step")
    ap.add_argument("--e2e-depth", type=int, default=6,
                    help="device input sets of the end-to-end loop (copies run up to depth-1 steps "
                         "ahead, so a stall of the host link shorter than that many steps is "
                         "absorbed)")
    ap.add_argument("--e2e-copy", choices=("auto", "sm", "sm1", "ce"), default="auto",
                    help="end-to-end input copies: sm = fpo_h2d_copy (SM loads of mapped pinned "
                         "memory) in one part per long GEMM phase of the error signal, started "
                         "as the phase begins; sm1 = one fpo_h2d_copy per step; ce = "
                         "cudaMemcpyAsync per tensor; auto = sm when one step's copy, timed "
                         "alone, is shorter than those GEMM phases, else sm1")
    ap.add_argument("--band", type=int, default=0,
                    help="GEMM rasterisation band height in tiles (0: library default; tuning)")
    ap.add_argument("--gemm-variant", type=int, choices=(-1, 0, 1, 2), default=-1,
                    help="tensor-core GEMM kernel: 0 single-CTA tiles, 1 CTA-pair tiles, "
                         "2 CTA-pair tiles with a 256x512 projection, -1 library default")
    ap.add_argument("--window-stress", action="store_true",
                    help="+-1 hidden states and W_U x 64: most tokens fall outside the direct "
                         "algorithm's anchor window (its worst case); reports the rows recomputed")
    ap.add_argument("--shape", default=None,
                    help="T,d,d_ff,V,layers override of the workload's shape (small ncu cases)")
    ap.add_argument("--cpu-tokens", type=int, default=256,
                    help="tokens of the oracle sample behind cpu_baseline (~10 s of CPU work "
                         "at the OLMo shape on 16 cores)")
    ap.add_argument("--ref-tokens", type=int, default=0,
                    help="tokens of the oracle sample of each --impl reference step (0: one to "
                         "four per host thread, fewer for longer runs, so that every core works "
                         "and the run stays within a few minutes)")
    ap.add_argument("--no-cpu", action="store_true", help="skip the oracle CPU baseline")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end run")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")

    if args.impl != "reference":  # the oracle arm neither builds nor loads libfpo
        ensure_built()
    from synth import WORKLOADS  # noqa: E402
    wl = WORKLOADS[args.workload]
    if args.shape:
        import dataclasses
        T, d, d_ff, V, L = (int(x) for x in args.shape.split(","))
        wl = dataclasses.replace(wl, name=f"{wl.name}@{T}x{d}x{d_ff}x{V}x{L}", T=T, d=d, d_ff=d_ff,
                                 V=V, layers=L)
    if args.impl == "reference":
        run_reference(args, wl)
    else:
        run_fpo(args, wl)


if __name__ == "__main__":
    main()

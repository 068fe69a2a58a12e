"""Batch-1 decode throughput of self-speculative decoding with the LEDE policy
on a synthetic Llama-2-7B-shaped decoder (bf16, prompt 512, 256 new tokens),
beside plain GPU autoregressive decoding and static (l, k) speculation on the
same kernels.

One step = one generation of the workload's new tokens through the whole hot
path (walk, drafting, verification, acceptance, rollback), timed with CUDA
events on the engine's stream after an untimed prefill.  Weights (13.5 GB)
are larger than L2, so no flush is needed between steps.

Prints one JSON line.  --impl reference times the CPU oracle instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

REPO = os.path.dirname(os.path.abspath(__file__))
if REPO not in sys.path:
    sys.path.insert(0, REPO)

import numpy as np  # noqa: E402

import synth  # noqa: E402
from synth.workloads import WORKLOADS  # noqa: E402

METRIC = "batch-1 decode tokens/sec and % of HBM-bandwidth roofline vs GPU AR/static"
CLOCK_FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


SAMPLE_SEED = 7  # uniforms of the sampled-decoding comparison lines
NOMINAL_HBM_GBS = 8000.0  # GB300 HBM3e, nominal (the measured copy bandwidth is the peak used)


def measured_peaks() -> dict:
    p = os.path.join(REPO, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm_gbs=float(d["hbm_gbs"]), src="measured")
    return dict(hbm_gbs=6800.0, src="fallback")


# DRAM traffic of the dominant kernel from the committed ncu summaries: valid
# only while the kernel's sources are the ones that were captured.
TRAFFIC_PROFILES = {"k_chain(o+gate_up+down+next_qkv)": "k_chain_llama2-7b.md"}
TRAFFIC_SOURCES = ("tile.cu", "tc.cuh", "pipe.cuh", "headpart.cuh")


def measured_traffic(kernel: str) -> int | None:
    """DRAM read + write bytes per single-row launch of `kernel` on the
    Llama-2-7B shape from one ncu capture, or None when there is no summary
    or the kernel sources no longer hash to the captured value."""
    name = TRAFFIC_PROFILES.get(kernel)
    if name is None:
        return None
    try:
        text = open(os.path.join(REPO, "profiles", name)).read()
        h = hashlib.sha256()
        for f in TRAFFIC_SOURCES:
            with open(os.path.join(REPO, "paper_2606_03113_gb300", "csrc", f), "rb") as fh:
                h.update(fh.read())
    except OSError:
        return None
    digest = re.search(r"`([0-9a-f]{64})`", text)
    nbytes = re.search(r"dram bytes per launch \(M = 1\): (\d+)", text)
    if not digest or not nbytes or digest.group(1) != h.hexdigest():
        return None
    return int(nbytes.group(1))


# --------------------------------------------------------------- bytes model

def round_bytes(w, tr: dict) -> float:
    """HBM bytes the method must read in one round: for each visited
    candidate the LM head, the layers up to l* once for the pending token,
    (k - 1) further drafts through l* layers + head, and the full model +
    head for verification; KV reads of every layer pass at its context."""
    s = w.shape
    Wl, head = s.layer_weight_bytes(), s.lm_head_bytes()
    kvpl = s.kv_bytes_per_pos_layer()
    L, pos = s.n_layers, tr["pos"]
    b = 0.0
    if tr["kcap"] > 0:
        l_star, k = tr["lstar"], tr["k"]
        b += len(tr["visited"]) * head + l_star * (Wl + kvpl * (pos + 1))
        for i in range(1, k):
            b += l_star * (Wl + kvpl * (pos + i + 1)) + head
    k = tr["k"]
    b += L * (Wl + kvpl * (pos + k + 1)) + head
    return b


def kernels_in_round(w, tr: dict) -> int:
    from paper_2606_03113_gb300.runtime import kernels_per_round
    return kernels_per_round(tr, w.shape.n_layers, 0, bf16=w.shape.dtype == "bf16")


# ------------------------------------------------------------------ clocks

class ClockSampler:
    def __init__(self, device_index: int):
        self.idx = device_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={CLOCK_FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
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
                f = [x.strip() for x in line.split(",")]
                if len(f) >= 9:
                    rows.append(f)
            os.unlink(self.path)
        if not rows:
            return dict(sm_mhz=None, sm_max_mhz=None, reasons=["unavailable"], samples=0)
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        reasons = set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            for name, v in zip(names, r[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        return dict(sm_mhz=statistics.median(sm) if sm else None,
                    sm_max_mhz=max(mx) if mx else None, reasons=sorted(reasons),
                    samples=len(rows))


# --------------------------------------------------------------- oracle arm

def oracle_sample(w, n_prompt: int, n_new: int, policy: str, om=None) -> dict:
    """Times the CPU oracle (as it stands) on a bounded sample of the
    workload: prefill of the first n_prompt prompt tokens, then n_new decoded
    tokens; the decode rate is the reported number."""
    import oracle
    t0 = time.perf_counter()
    om = om or oracle.Model(w.shape)
    t_model = time.perf_counter() - t0
    ids = synth.prompt_ids(n_prompt, w.shape.vocab)
    s = om.session(n_prompt + n_new + w.kmax + 2)
    s.prefill(ids)
    if policy == "ar":
        P = oracle.make_policy(oracle.POLICY_AR)
    else:
        P = oracle.make_policy(oracle.POLICY_LEDE, w.candidates, kmax=w.kmax,
                               q_params=synth.qnet_hidden_params(3, w.qnet_hidden),
                               q_hidden=w.qnet_hidden)
    t1 = time.perf_counter()
    out, logs = s.generate(P, n_new)
    dt = time.perf_counter() - t1
    return dict(value=n_new / dt, seconds=dt, model_seconds=t_model, cores=oracle.num_threads(),
                model=om,
                sample=f"{w.name}-shaped oracle (fp64), {policy} policy: prefill of the first "
                       f"{n_prompt} prompt tokens (untimed), then {n_new} decoded tokens timed")


def run_reference(args, w, rank: int, world: int):
    if rank != 0:
        return
    steps = []
    samples = None
    om = None
    for i in range(args.warmup + args.steps):
        r = oracle_sample(w, args.ref_prompt, args.ref_new, args.policy, om)
        om = r["model"]
        if i >= args.warmup:
            steps.append(r)
        samples = r
    tok = args.ref_new * len(steps)
    sec = sum(r["seconds"] for r in steps)
    value = tok / sec
    line = dict(metric=METRIC, value=value, unit="tokens/s", n_gpus=world, steps=args.steps,
                warmup=args.warmup, ms_per_step=1e3 * sec / len(steps), higher_is_better=True,
                scaling="weak", vs_baseline=None, dtype="f64", data="synthetic", impl="reference",
                config=dict(workload=f"{w.name}-shaped decoder, batch 1, {args.policy} policy",
                            sample=samples["sample"]),
                cpu_baseline=dict(value=value, unit="tokens/s", cores=samples["cores"],
                                  kind="oracle", sample=samples["sample"]),
                e2e=dict(value=value, unit="tokens/s", h2d_bytes_per_step=0,
                         d2h_bytes_per_step=0))
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------- replicas

def aggregate_replicas(local_ms: float, local_tokens: float, device: str = "cpu") -> tuple:
    """Whole-job timing of N independent replicas (one sequence per rank, no
    data-path collective): the slowest rank's time and the tokens of all
    ranks.  A no-op without an initialised process group of size > 1."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1):
        return float(local_ms), float(local_tokens)
    mx = torch.tensor([float(local_ms)], dtype=torch.float64, device=device)
    tot = torch.tensor([float(local_tokens)], dtype=torch.float64, device=device)
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(tot, op=dist.ReduceOp.SUM)
    return float(mx[0]), float(tot[0])


# ------------------------------------------------------------------ GPU arm

def time_generate(eng, ids, n_new, dist_barrier) -> tuple:
    import torch
    eng.prefill(ids)
    dist_barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(eng.stream)
    eng.generate_async(n_new)
    e1.record(eng.stream)
    nr, ne, tr = eng.generate_result(traces=True, cap=n_new)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1), ne, tr


def static_grid(w, set_policy, eng, ids, n_new, barrier, n_grid: int = 64, top: int = 3) -> dict:
    """Best static (l, k) (LayerSkip's fixed exit layer and draft length,
    §4.1 Baselines): every candidate exit layer x every draft length 1..kmax
    timed on a short generation of n_grid tokens, then the `top` fastest
    points again on the full n_new tokens; the best of those is reported."""
    pts = []
    for l in w.candidates:
        for k in range(1, w.kmax + 1):
            set_policy("static", l, k)
            time_generate(eng, ids, 8, barrier)
            r = time_generate(eng, ids, n_grid, barrier)
            pts.append((r[1] / (r[0] / 1e3), l, k))
    pts.sort(reverse=True)
    best = None
    for _, l, k in pts[:top]:
        set_policy("static", l, k)
        time_generate(eng, ids, n_new, barrier)
        r = time_generate(eng, ids, n_new, barrier)
        tr = r[2]
        cand = dict(tok_s=r[1] / (r[0] / 1e3), l=l, k=k,
                    acc_rate=sum(t["a"] for t in tr) / max(1, sum(t["k"] for t in tr)),
                    gb_per_token=sum(round_bytes(w, t) for t in tr) / r[1] / 1e9)
        if best is None or cand["tok_s"] > best["tok_s"]:
            best = cand
    best["grid"] = (f"l in {list(w.candidates)} x k in 1..{w.kmax}: {len(pts)} points timed on "
                    f"{n_grid} new tokens, the {top} fastest again on {n_new}")
    best["grid_top"] = [dict(l=l, k=k, tok_s=round(t, 1)) for t, l, k in pts[:8]]
    return best


KERNEL_NAMES = {0: "k_qkv", 1: "k_attn", 2: "k_resid(wo)", 3: "k_gate_up",
                4: "k_resid(w_down)", 5: "k_head", 6: "k_chain(o+gate_up+down+next_qkv)"}


def kernel_roofline(eng, w, peak: float, pos0: int, iters: int = 5, graphs: bool = True) -> dict:
    """Live CUDA-event timing, on the engine's stream where the kernels are
    launched, of each hot-path kernel of a single-row pass: one launch per
    layer over all layers (so a launch never finds its weights in L2),
    replayed from a CUDA graph so host launch cost does not enter.  Bytes are
    the algorithmic ones: the launch's weight matrix; attention counts its
    K/V reads at context pos0."""
    import torch
    s = w.shape
    L = s.n_layers
    elt = s.elt_bytes
    qd = s.n_heads * s.head_dim
    byts = {0: s.qkv_rows * s.d_model * elt, 1: s.kv_bytes_per_pos_layer() * (pos0 + 1),
            2: s.d_model * qd * elt, 3: 2 * s.ffn_dim * s.d_model * elt,
            4: s.d_model * s.ffn_dim * elt, 5: s.vocab * s.d_model * elt}
    kerns = (0, 1, 2, 3, 4, 5)
    if s.dtype == "bf16":
        # the chained launch the layer passes use: O, gate/up, down of layer
        # l and the QKV of layer l + 1 (the last layer has no QKV phase)
        byts[6] = byts[2] + byts[3] + byts[4] + byts[0] * (L - 1) / L
        kerns = kerns + (6,)
    out = {}
    st = eng.stream
    for kern in kerns:
        layers = [0] * 8 if kern == 5 else list(range(L))

        def run():
            for l in layers:
                eng.op_layer(kern, l, 1, pos0)

        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        run()
        torch.cuda.synchronize()
        if graphs:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=st):
                run()
            with torch.cuda.stream(st):  # replay() launches on the current stream
                g.replay()
                torch.cuda.synchronize()
                e0.record(st)
                for _ in range(iters):
                    g.replay()
                e1.record(st)
        else:
            e0.record(st)
            for _ in range(iters):
                run()
            e1.record(st)
        torch.cuda.synchronize()
        us = e0.elapsed_time(e1) * 1e3 / (iters * len(layers))
        b = byts[kern]
        out[KERNEL_NAMES[kern]] = dict(us=us, bytes=b, launches_per_forward=1 if kern == 5 else L,
                                       gbs=b / us / 1e3, frac=b / us / 1e3 / peak)
    return out


def verify_rows_probe(eng, w, ids, layers, rows, iters: int = 20) -> dict:
    """Time of a pass over layers 1..l (embedding, the layers, one exit head)
    for M rows at the end of the prompt, for each l and M: CUDA events on the
    engine's stream, mean of `iters` passes after one warm-up.  The difference
    t(l, k + 1) - t(l, 1) bounds what reusing the drafts' early-layer states
    in verification (LayerSkip's verify reuse) could save per round: the
    layers' weights are read once for any M, so only the per-row work and the
    KV writes of the k drafted rows in layers 1..l* would go."""
    import torch
    from paper_2606_03113_gb300 import ssd as S
    out = {}
    n0 = len(ids) - max(rows)
    eng.set_ar()
    eng.prefill(ids[:n0])
    for l in layers:
        out[l] = {}
        for M in rows:
            toks = ids[n0:n0 + M]
            S.ssd_forward_exit(eng.ctx, toks, n0, l, 5, False, w.shape.vocab)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            e0.record(eng.stream)
            for _ in range(iters):
                S.ssd_forward_exit(eng.ctx, toks, n0, l, 5, False, w.shape.vocab)
            e1.record(eng.stream)
            torch.cuda.synchronize()
            out[l][M] = e0.elapsed_time(e1) * 1e3 / iters
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama2-7b", choices=sorted(WORKLOADS))
    ap.add_argument("--policy", default="lede", choices=["lede", "ar", "static"])
    ap.add_argument("--qnet", default="trained", choices=["trained", "seeded"],
                    help="LEDE Q-network: trained offline by DQN on experience from this model "
                         "(outside the timed region), or the seeded random network")
    ap.add_argument("--train-prompts", type=int, default=4)
    ap.add_argument("--train-gen", type=int, default=128)
    ap.add_argument("--train-episodes", type=int, default=30000)
    ap.add_argument("--save-exit-table", default="",
                    help="write the Q-network's training experience to this .npz file")
    ap.add_argument("--gen", type=int, default=0, help="new tokens per step (default: workload)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-compare", action="store_true", help="skip the AR / static lines")
    ap.add_argument("--no-static-grid", action="store_true",
                    help="skip the sweep of every static (l, k) for the best static setting")
    ap.add_argument("--ref-prompt", type=int, default=16)
    ap.add_argument("--ref-new", type=int, default=4)
    ap.add_argument("--kernels-only", action="store_true",
                    help="prefill, then launch each hot-path kernel eagerly over all layers "
                         "(for per-kernel ncu captures) and print their timings")
    ap.add_argument("--verify-rows", action="store_true",
                    help="time passes over layers 1..l for 1..kmax+1 rows (the per-round saving "
                         "bound of reusing drafted rows' early layers in verification) and exit")
    ap.add_argument("--layers", type=int, default=0,
                    help="override the layer count (small cases for ncu --set full)")
    args = ap.parse_args()

    w = WORKLOADS[args.workload]
    if args.layers:
        from dataclasses import replace
        w = replace(w, shape=replace(w.shape, n_layers=args.layers,
                                     name=f"{w.shape.name}-{args.layers}l"),
                    candidates=tuple(c for c in w.candidates if c < args.layers) or (1,))
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        run_reference(args, w, rank, world)
        return

    import torch
    import torch.distributed as dist
    if world > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)

    def barrier():
        if world > 1:
            dist.barrier()

    from paper_2606_03113_gb300.runtime import DeviceModel, Engine
    peaks = measured_peaks()
    peak = peaks["hbm_gbs"]
    n_new = args.gen or w.gen_len
    model = DeviceModel(w.shape, f"cuda:{local}")
    stream = torch.cuda.Stream(device=local)
    eng = Engine(model, w.max_seq, stream=stream)
    ids = synth.prompt_ids(w.prompt_len, w.shape.vocab)

    seeded_qp = synth.qnet_hidden_params(3, w.qnet_hidden)
    qnet_info = dict(kind="seeded")
    qp = seeded_qp
    if args.policy == "lede" and args.qnet == "trained" and not args.kernels_only:
        # offline DQN (§3.2) on exit statistics of this model's own greedy
        # continuations of prompts other than the benchmark's
        from paper_2606_03113_gb300 import policy as PL
        t0 = time.perf_counter()
        prompts = [synth.prompt_ids(128, w.shape.vocab, seed=synth.SEED_PROMPT + 1 + i)
                   for i in range(args.train_prompts)]
        table = PL.collect_exit_table(eng, w.candidates, prompts, args.train_gen)
        if args.save_exit_table and rank == 0:
            table.save(args.save_exit_table)
        t1 = time.perf_counter()
        qp, walk, tlog = PL.train_policy(table, w.qnet_hidden, episodes=args.train_episodes)
        t2 = time.perf_counter()
        qnet_info = dict(kind="trained (offline DQN)", positions=int(table.n),
                         exit_agreement={int(c): round(float(a), 3)
                                         for c, a in zip(w.candidates, table.agreement())},
                         walk_return=round(walk["mean_return"], 4),
                         walk_exit_layer=round(walk["exit_layer"], 2),
                         hindsight_return=round(PL.oracle_walk_return(table), 4),
                         separation_auc_conf={int(c): (round(v["conf"], 3)
                                                       if np.isfinite(v["conf"]) else None)
                                              for c, v in table.separation().items()},
                         updates=tlog.updates, collect_s=round(t1 - t0, 1),
                         train_s=round(t2 - t1, 1))

    def set_policy(kind, l=0, k=0, q=None, temperature=0.0):
        smp = dict(temperature=temperature, sample_seed=SAMPLE_SEED)
        if kind == "ar":
            eng.set_ar(**smp)
        elif kind == "static":
            eng.set_static(l, k, kmax=w.kmax, **smp)
        else:
            eng.set_lede(w, qp if q is None else q, **smp)

    L = w.shape.n_layers
    if args.verify_rows:
        lays = sorted({c for c in w.candidates} | {L})
        rows = sorted({1, 2, 4, 8, min(w.kmax + 1, 17)})
        r = verify_rows_probe(eng, w, ids, lays, rows)
        if rank == 0:
            print(json.dumps(dict(verify_rows_us=r, workload=w.name, context=len(ids))), flush=True)
        eng.close()
        return
    if args.kernels_only:
        eng.set_ar()
        eng.prefill(ids)
        roof = kernel_roofline(eng, w, peak, pos0=w.prompt_len, iters=3, graphs=True)
        if rank == 0:
            print(json.dumps(dict(kernels=roof, workload=w.name, peak=peak)), flush=True)
        eng.close()
        return
    static_lk = (max(1, L // 4), 4)  # the LayerSkip-style default (E = L/4, d = 4)
    set_policy(args.policy, *static_lk)
    for _ in range(args.warmup):
        time_generate(eng, ids, n_new, barrier)
    results = []
    with ClockSampler(local) as clk:
        for _ in range(args.steps):
            results.append(time_generate(eng, ids, n_new, barrier))
    clocks = clk.summary()
    ms = [r[0] for r in results]
    toks = [r[1] for r in results]
    local_ms = sum(ms)
    total_ms, total_tok = aggregate_replicas(local_ms, float(sum(toks)), f"cuda:{local}")
    value = total_tok / (total_ms / 1e3)
    traces = results[-1][2]
    bytes_step = sum(round_bytes(w, tr) for tr in traces)
    step_gbs = bytes_step / (results[-1][0] / 1e3) / 1e9
    launches = sum(sum(kernels_in_round(w, tr) for tr in r[2]) for r in results)
    acc_k = sum(tr["k"] for tr in traces)
    policy_stats = dict(rounds=len(traces), E=float(np.mean([t["lstar"] for t in traces if t["kcap"] > 0]
                                                            or [0])),
                        d=acc_k / max(1, sum(1 for t in traces if t["kcap"] > 0)),
                        acc_rate=sum(t["a"] for t in traces) / max(1, acc_k),
                        tokens_per_round=n_new / max(1, len(traces)),
                        rounds_multi_draft=sum(1 for t in traces if t["k"] > 1),
                        gb_per_token=bytes_step / n_new / 1e9)

    # e2e through the public API with host buffers: prompt in, tokens out
    from paper_2606_03113_gb300 import ssd as S
    t0 = time.perf_counter()
    S.ssd_prefill(eng.ctx, ids)
    out, _, _ = S.ssd_generate(eng.ctx, n_new)
    e2e_s = time.perf_counter() - t0
    e2e = dict(value=n_new / e2e_s, unit="tokens/s", h2d_bytes_per_step=int(ids.nbytes),
               d2h_bytes_per_step=int(out.nbytes),
               note="ssd_prefill (host prompt) + ssd_generate (host tokens), wall clock")

    roof = kernel_roofline(eng, w, peak, pos0=w.prompt_len + n_new // 2)
    # the dominant kernel among those a forward pass launches (bf16: the
    # chained launch replaces the per-matrix ones)
    launched = {k: v for k, v in roof.items()
                if KERNEL_NAMES[6] not in roof or k in (KERNEL_NAMES[6], "k_attn", "k_head")}
    dom = max(launched.items(), key=lambda kv: kv[1]["us"] * kv[1]["launches_per_forward"])
    traffic = measured_traffic(dom[0]) if w.name == "llama2-7b" else None
    roofline = dict(bound="hbm", achieved=dom[1]["gbs"], peak=peak, unit="GB/s",
                    frac=dom[1]["gbs"] / peak, traffic=traffic,
                    frac_vs_nominal=dom[1]["gbs"] / NOMINAL_HBM_GBS,
                    kernel=f"{dom[0]} single-row ({dom[1]['bytes'] / 1e6:.1f} MB per launch)",
                    peak_source=f"{peaks['src']} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)",
                    kernels=roof,
                    decode_step=dict(achieved=step_gbs, frac=step_gbs / peak,
                                     frac_vs_nominal=step_gbs / NOMINAL_HBM_GBS,
                                     what="weight + KV bytes the round structure must read / step time"))

    compare = {}
    if not args.no_compare and args.policy == "lede":
        runs = [("ar", "ar", (0, 0), None, 0.0),
                ("static_layerskip", "static", static_lk, None, 0.0),
                ("static_l16_k4", "static", (L // 2, 4), None, 0.0),
                ("static_l24_k2", "static", (3 * L // 4, 2), None, 0.0)]
        if qnet_info["kind"] != "seeded":
            runs.append(("lede_seeded_qnet", "lede", (0, 0), seeded_qp, 0.0))
        # sampled decoding at the paper's language-modelling temperature
        runs += [("ar_sampled_t0.6", "ar", (0, 0), None, 0.6),
                 ("lede_sampled_t0.6", "lede", (0, 0), None, 0.6)]
        for name, kind, lk, q, temp in runs:
            set_policy(kind, *lk, q=q, temperature=temp)
            time_generate(eng, ids, n_new, barrier)
            r = time_generate(eng, ids, n_new, barrier)
            tr = r[2]
            compare[name] = dict(tok_s=r[1] / (r[0] / 1e3), l=lk[0], k=lk[1],
                                 acc_rate=sum(t["a"] for t in tr) / max(1, sum(t["k"] for t in tr)),
                                 gb_per_token=sum(round_bytes(w, t) for t in tr) / r[1] / 1e9)
            if temp > 0:
                compare[name]["temperature"] = temp
        if not args.no_static_grid:
            compare["static_best"] = static_grid(w, set_policy, eng, ids, n_new, barrier)
        ar_bytes = L * w.shape.layer_weight_bytes() + w.shape.lm_head_bytes()
        compare["ar_roofline_tok_s"] = peak * 1e9 / ar_bytes

    cpu = None
    if rank == 0 and not args.no_cpu_baseline and world == 1:
        r = oracle_sample(w, args.ref_prompt, args.ref_new, args.policy)
        cpu = dict(value=r["value"], unit="tokens/s", cores=r["cores"], kind="oracle",
                   sample=r["sample"])

    line = dict(metric=METRIC, value=value, unit="tokens/s", n_gpus=world, steps=args.steps,
                warmup=args.warmup, ms_per_step=total_ms / args.steps, higher_is_better=True,
                scaling="weak", vs_baseline=None, dtype="bf16", data="synthetic",
                config=dict(workload=f"{w.name}-shaped decoder (random-init bf16), batch 1, "
                                     f"prompt {w.prompt_len}, {n_new} new tokens per step, "
                                     f"{args.policy} policy"
                                     + ((" (" + qnet_info["kind"] + " Q-network)")
                                        if args.policy == "lede" else ""),
                            l2="inputs larger than L2 (13.5 GB of weights streamed per pass)",
                            parallelism=f"replicas x{world}" if world > 1 else "single GPU"),
                roofline=roofline, cpu_baseline=cpu, e2e=e2e, gpu_launches=launches,
                clocks=clocks, policy_stats=policy_stats, qnet=qnet_info, compare=compare)
    if rank == 0:
        print(json.dumps(line), flush=True)
    eng.close()
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()

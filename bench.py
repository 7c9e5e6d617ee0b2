#!/usr/bin/env python
"""Throughput of the DVI decode step + online drafter update on GB300.

One bench step = `update_every` draft_verify_commit calls (K draft passes
through layers 1..k and the drafter head, one verify pass of the K rows
through layers k+1..L and the LM head, accept / commit / rollback / log)
plus one drafter update on the logged buffer -- every row of the hot path.
Default workload: Llama-2-7B-shaped decoder in bf16, batch 1, split k=2
(the paper's split), k_spec 5, 1024-token Zipf(1.1) prompt, update every 4
steps under the KL->RL schedule; random-init weights (synthetic, seeded).

    python bench.py [--gpus N --steps K --warmup W] [--impl reference]

Multi-GPU runs are independent replicas (one process per GPU, no
collective on the data path); value = tokens committed by all ranks / the
slowest rank's time.  `--impl reference` times the CPU oracle instead (rank 0).
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from workloads import workload, make_weights, make_prompts  # noqa: E402

METRIC = "committed tokens/s at batch 1"
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return dict(PEAKS_FALLBACK), "fallback"


# ---------------------------------------------------------------- byte model
def layer_bytes(s, esz):
    nq, nkv = s.n_heads * s.head_dim, s.n_kv_heads * s.head_dim
    return (nq * s.d_model + 2 * nkv * s.d_model + s.d_model * nq + 3 * s.d_model * s.d_ffn) * esz


def kv_row_bytes(s, esz):
    return 2 * s.n_kv_heads * s.head_dim * esz


def step_bytes(w, n_ctx):
    """Algorithmic HBM bytes of one decode step at committed lengths n_ctx[b].

    Weights are streamed once per pass; every KV row a pass attends to is
    read once for all its queries.  Returns (draft bytes, verify bytes).
    """
    s, esz, k, K = w.shape, (2 if w.dtype == "bf16" else 4), w.split_k, w.k_spec
    lb, kvb, head = layer_bytes(s, esz), kv_row_bytes(s, esz), s.vocab * s.d_model * esz
    lora = (s.vocab + s.d_model) * w.lora_rank * 4
    draft = K * (k * lb + head + lora)
    verify = (s.n_layers - k) * lb + head
    for n in n_ctx:
        draft += sum(k * (n + j + 1) * kvb for j in range(K))
        verify += (s.n_layers - k) * (n + K) * kvb
    return draft, verify


def update_bytes(w, rows):
    """Algorithmic HBM bytes of one LoRA drafter update on `rows` buffer rows:
    the logged drafter logits z and verifier logits (rows x V f32 each) and
    head inputs u (bf16 hi/lo or f32), and A, B with their Adam moments read
    and written plus their gradients written.  W^S is not read: z was logged
    by the drafter head while drafting."""
    s = w.shape
    usz = 4  # bf16 hi + lo planes, or one f32 plane
    lora = (s.vocab + s.d_model) * w.lora_rank * 4
    return 2 * rows * s.vocab * 4 + rows * s.d_model * usz + 7 * lora


def prefill_flops(w, n):
    """Algorithmic FLOPs of prefilling one n-token prompt: 2 per weight per
    token for every layer's projections, the causal attention's two
    products (2 x hd per query head and attended position, the query's own
    position included), and the LM head on the last row."""
    s = w.shape
    params = layer_bytes(s, 1)
    attended = n * (n + 1) // 2
    per_layer = 2 * params * n + 2 * 2 * s.n_heads * s.head_dim * attended
    return s.n_layers * per_layer + 2 * s.vocab * s.d_model


def prefill_bytes(w, n, chunk):
    """HBM bytes of prefilling one n-token prompt in passes of `chunk` rows,
    as this library runs it: every pass streams all L layers' weights once,
    reads the K/V rows of its prefix (its own included) once per layer and
    writes its own; the LM head runs on the last row only.  With chunk = n
    (one pass over the whole prompt) this is the algorithm's own minimum."""
    s, esz = w.shape, (2 if w.dtype == "bf16" else 4)
    lb, kvb = layer_bytes(s, esz), kv_row_bytes(s, esz)
    total = s.vocab * s.d_model * esz
    for c0 in range(0, n, chunk):
        rows = min(chunk, n - c0)
        total += s.n_layers * (lb + (c0 + rows) * kvb + rows * kvb)
    return total


def prefill_alg_bytes(w, n):
    """Algorithmic HBM bytes of an n-token prefill: every weight once, every
    K/V row written once and read once."""
    return prefill_bytes(w, n, n)


def measured_traffic(w, n_attended, persistent=False):
    """Per-launch DRAM traffic of the verify pass from the committed ncu summary.

    The summary holds the bytes ncu counted per deep layer's projections (or,
    for the persistent chain, per chain launch), the LM head, and one deep
    layer's attention at a given number of 64-position chunks; the pass's
    traffic is scaled to this workload's layer count and context.  Returns
    None when no capture matches the workload.
    """
    p = os.path.join(ROOT, "profiles", "verify_pass_dram_7b_width.md")
    if not os.path.exists(p):
        return None
    m = None
    key = "traffic-model-persistent:" if persistent else "traffic-model:"
    for ln in open(p):
        if ln.startswith(key):
            m = json.loads(ln.split(":", 1)[1])
    s = w.shape
    if m is None or (m["d_model"], m["n_heads"], m["d_ffn"], m["vocab"]) != (s.d_model, s.n_heads, s.d_ffn,
                                                                             s.vocab) \
            or m["dtype"] != w.dtype or m["batch"] != w.batch or m["k_spec"] != w.k_spec:
        return None
    deep = w.shape.n_layers - w.split_k
    chunks = float(np.mean([-(-int(round(n + w.k_spec)) // 64) * 64 for n in n_attended]))
    attn = deep * m["attn_bytes_per_deep_layer"] * chunks / m["attn_chunk_positions"]
    if persistent:
        return (m["qkv_first_bytes"] + (deep - 1) * m["chain_bytes_per_deep_layer"] + m["chain_last_bytes"]
                + m["head_bytes"] + attn)
    return deep * m["proj_bytes_per_deep_layer"] + attn + m["head_bytes"]


def prefill_roofline(flops, alg_bytes, ms, pk, traffic=None):
    """The prefill against the roofline that bounds the algorithm: its FLOPs
    over the burst bf16 tensor throughput, or its algorithmic bytes over the
    copy bandwidth, whichever takes longer at peak.  `traffic` (the bytes the
    implementation moves, weights re-read per pass included) is reported
    beside it, not used for the fraction."""
    t_hbm = alg_bytes / (pk["hbm_gbs"] * 1e9)
    t_tc = flops / (pk["bf16_tflops"] * 1e12)
    if t_tc >= t_hbm:
        ach = flops / (ms / 1e3) / 1e12
        r = {"bound": "tensor", "achieved": ach, "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
             "frac": ach / pk["bf16_tflops"]}
    else:
        ach = alg_bytes / (ms / 1e3) / 1e9
        r = {"bound": "hbm", "achieved": ach, "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": ach / pk["hbm_gbs"]}
    r.update({"flops": flops, "alg_bytes": alg_bytes, "traffic_model": traffic})
    return r


# ---------------------------------------------------------------- clocks
class ClockSampler:
    REASONS = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, gpu_index):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--query-gpu={q}", "--format=csv,noheader,nounits",
                                       "-i", str(gpu_index), "-lms", "25"], stdout=self.f,
                                      stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None

    def stop(self):
        if self.p is None:
            return None
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.p.kill()
        self.f.flush()
        self.f.seek(0)
        rows = [r.split(",") for r in self.f.read().strip().splitlines() if r.strip()]
        os.unlink(self.f.name)
        sm, mx, reasons = [], 0.0, set()
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx = max(mx, float(r[2]))
            except (ValueError, IndexError):
                continue
            for name, val in zip(self.REASONS, r[5:9]):
                if val.strip().lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------- CPU oracle
class OracleRun:
    """The CPU oracle (numpy float32) on the workload's first prompt, at the
    workload's own context: the whole prompt is prefilled once (untimed),
    then DVI steps (with the drafter update every `update_every` steps) and
    greedy AR steps are timed on the host cores in bounded samples."""

    def __init__(self, w, W, room=1024):
        from oracle import OracleModel, DrafterUpdater
        from oracle.decode import prefill
        self.w = w
        self.m = OracleModel(W, w.shape, w.lora_gamma, dtype=np.float32)
        self.upd = DrafterUpdater(self.m, w.update)
        P = make_prompts(w)[0]
        self.prompt = len(P)
        self.cache = self.m.new_cache(len(P) + room)
        t0 = time.perf_counter()
        self.tok, _ = prefill(self.m, self.cache, P)
        self.prefill_s = time.perf_counter() - t0
        self.n, self.buf, self.steps = len(P), [], 0

    def room(self, rows):
        return self.n + rows + 1 <= self.cache.max_len

    def dvi(self, budget_s, steps_cap=None):
        """DVI steps until `budget_s` has passed at an update boundary (or the
        cache is full): (tokens committed, steps, seconds)."""
        from oracle.decode import dvi_step
        w, committed, steps = self.w, 0, 0
        t0 = time.perf_counter()
        while self.room(w.k_spec):
            fields, tuples, self.n, self.tok = dvi_step(self.m, self.cache, self.n, self.tok, w.split_k, w.k_spec)
            committed += len(fields[3])
            self.buf.extend(tuples)
            steps += 1
            self.steps += 1
            if self.steps % w.update_every == 0:
                self.upd.update(self.buf)
                self.buf = []
                if time.perf_counter() - t0 >= budget_s or (steps_cap and steps >= steps_cap):
                    break
        return committed, steps, time.perf_counter() - t0

    def ar(self, budget_s):
        """Greedy AR steps of the full model until `budget_s` has passed:
        (tokens, seconds)."""
        from oracle.decode import ar_step
        n_tok = 0
        t0 = time.perf_counter()
        while self.room(1) and (n_tok == 0 or time.perf_counter() - t0 < budget_s):
            self.tok, _ = ar_step(self.m, self.cache, self.n, self.tok)
            self.n += 1
            n_tok += 1
        return n_tok, time.perf_counter() - t0


def cpu_baseline_dict(run, dvi, ar, cores):
    c, st, sec = dvi
    ntok, asec = ar
    w = run.w
    v, v_ar = c / sec, ntok / asec
    return {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "ar_tokens_per_s": v_ar, "dvi_over_ar": v / v_ar,
            "sample": (f"{w.shape.n_layers}-layer d{w.shape.d_model} decoder in numpy float32 on the "
                       f"{run.prompt}-token prompt (prefill untimed, {run.prefill_s:.0f} s), {st} DVI steps "
                       f"with an update every {w.update_every} in {sec:.1f} s, then {ntok} greedy AR steps "
                       f"in {asec:.1f} s")}


# ---------------------------------------------------------------- main
def combine_ranks(ms, committed, world):
    """Whole-job figures over replica ranks: the slowest rank's time and the
    tokens every rank committed (max and sum over the process group)."""
    if world <= 1:
        return ms, float(committed)
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms, float(committed)], dtype=torch.float64)
    tmax = t.clone()
    dist.all_reduce(tmax, op=dist.ReduceOp.MAX)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(tmax[0]), float(t[1])


def reference_arm(args, w, rank):
    """--impl reference: the oracle as it stands, timed on the host cores
    (rank 0 only) on the workload's own prompt: one untimed prefill, W
    warm-up samples, then K timed samples of about cpu_seconds / K each."""
    if rank != 0:
        return 0
    cores = os.cpu_count() or 1
    run = OracleRun(w, make_weights(w))
    run.dvi(0.0, steps_cap=args.warmup * w.update_every)
    per = max(1.0, args.cpu_seconds / max(1, args.steps))
    tot_c, tot_s, tot_steps = 0, 0.0, 0
    for _ in range(args.steps):
        c, st, sec = run.dvi(per)
        tot_c += c
        tot_s += sec
        tot_steps += st
    val = tot_c / tot_s
    line = {"impl": "reference", "metric": METRIC, "value": val, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_s / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": {"workload": w.name},
            "cpu_baseline": {"value": val, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": f"{args.steps} samples of ~{per:.1f} s: numpy float32 oracle on the "
                                       f"{run.prompt}-token prompt (prefill untimed, {run.prefill_s:.0f} s), "
                                       f"{tot_steps} DVI steps with updates"},
            "e2e": {"value": val, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def make_engine(w, dw, max_len, local, persistent=False, megakernel=True):
    from paper_2510_05421_gb300 import DVIEngine
    return DVIEngine(w.shape, w.dtype, dw, batch=w.batch, k_spec=w.k_spec, split_k=w.split_k,
                     lora_rank=w.lora_rank, lora_gamma=w.lora_gamma, max_seq_len=max_len,
                     log_steps=w.update_every, device=local, persistent=persistent, megakernel=megakernel)


def time_dvi(eng, w, hyper, warmup, steps, dev, world=1, clocks=False):
    """W warm-up and K timed bench steps (update_every decode steps + one
    drafter update each), CUDA events on the engine's stream."""
    import torch
    import torch.distributed as dist
    U = w.update_every

    def one_step():
        for _ in range(U):
            eng.step()
        eng.update(hyper)

    eng.log(True)
    for _ in range(warmup):
        one_step()
    eng.sync()
    lens0 = eng.buffer("LENS", torch.int32).cpu().numpy()
    st0 = eng.stats()
    eng.get_timing()
    eng.timing(True)
    sampler = ClockSampler(dev.index) if clocks else None
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(eng.stream)
    for _ in range(steps):
        one_step()
    e1.record(eng.stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    clk = sampler.stop() if sampler else None
    ms = e0.elapsed_time(e1)
    phases = eng.get_timing()
    eng.timing(False)
    st1 = eng.stats()
    lens1 = eng.buffer("LENS", torch.int32).cpu().numpy()
    dsteps = st1["steps"] - st0["steps"]
    return dict(ms=ms, committed=st1["committed"] - st0["committed"], decode_steps=dsteps,
                mat=(st1["accepted"] - st0["accepted"]) / max(1, dsteps * w.batch),
                launches=st1["kernel_launches"] - st0["kernel_launches"], phases=phases,
                lens0=lens0, lens1=lens1, clocks=clk, status=st1["device_flags"])


def time_ar(eng, dP, lens0, n_tokens, dev):
    """Greedy AR (dvi_ar_step, the speedup's denominator, Sec. 4.1) on the
    same engine, weights and context: every prompt prefilled again, advanced
    untimed to the context the timed DVI region started at, then enough AR
    steps for the same number of committed tokens, timed with CUDA events."""
    import torch
    B = len(dP)
    for b, p in enumerate(dP):
        eng.prefill(b, p)
    warm = max(3, int(round(float(np.mean([lens0[b] - len(dP[b]) for b in range(B)])))))
    for _ in range(warm):
        eng.ar_step()
    n_steps = max(1, -(-int(n_tokens) // B))
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(eng.stream)
    for _ in range(n_steps):
        eng.ar_step()
    e1.record(eng.stream)
    torch.cuda.synchronize(dev)
    ms = e0.elapsed_time(e1)
    return {"tokens_per_s": B * n_steps / (ms / 1e3), "ms_per_step": ms / n_steps, "steps": n_steps}


def update_roofline(w, u_ms, hbm):
    """The drafter update against its bytes (one update on a full buffer)."""
    rows = w.update_every * w.batch * w.k_spec
    nb = update_bytes(w, rows)
    ach = nb / (u_ms / 1e3) / 1e9
    return {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s", "frac": ach / hbm, "bytes": nb,
            "rows": rows, "note": "latency-bound: one cooperative launch, two grid barriers; W^S is not re-read"}


def pass_rooflines(w, r, hbm):
    """Draft- and verify-phase HBM fractions from the per-phase timing."""
    n_mid = (r["lens0"] + r["lens1"]) / 2.0
    draft_b, verify_b = step_bytes(w, n_mid)
    ph = r["phases"]
    v_ms = ph["verify"][0] / max(1, ph["verify"][1])
    d_ms = ph["draft"][0] / max(1, ph["draft"][1])
    u_ms = ph["update"][0] / max(1, ph["update"][1])
    return n_mid, draft_b, verify_b, d_ms, v_ms, u_ms


def extra_workload(name, args, local, dev, pk):
    """A second workload in the same run, reported beside the headline: the
    1B model's drafter and verifier often agree, so its stream exercises
    acceptance (mean accepted length, speedup over greedy AR)."""
    import torch
    from paper_2510_05421_gb300 import DeviceWeights, update_config
    w = workload(name)
    W = make_weights(w)
    dw = DeviceWeights.from_host(W, w.dtype, device=dev)
    P = make_prompts(w)
    U, K = w.update_every, w.k_spec
    steps = max(6, args.steps // 2)
    max_len = max(len(p) for p in P) + (args.warmup + steps) * U * K + 2 * K + 64
    eng = make_engine(w, dw, max_len, local, megakernel=not args.no_megakernel)
    dP = [torch.from_numpy(p).to(dev) for p in P]
    for b, p in enumerate(dP):
        eng.prefill(b, p)
    r = time_dvi(eng, w, update_config(w.update), args.warmup, steps, dev)
    ar = time_ar(eng, dP, r["lens0"], r["committed"], dev)
    eng.close()
    _, draft_b, verify_b, d_ms, v_ms, u_ms = pass_rooflines(w, r, pk["hbm_gbs"])
    value = r["committed"] / (r["ms"] / 1e3)
    return {"workload": w.name, "value": value, "unit": "tokens/s", "steps": steps,
            "decode_steps": r["decode_steps"], "mean_accepted_length": r["mat"],
            "ar_tokens_per_s": ar["tokens_per_s"], "speedup_vs_ar": value / ar["tokens_per_s"],
            "verify_frac": verify_b / (v_ms / 1e3) / 1e9 / pk["hbm_gbs"],
            "draft_frac": draft_b / (d_ms / 1e3) / 1e9 / pk["hbm_gbs"], "update_ms": u_ms,
            "device_flags": r["status"]}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=60)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="dvi", choices=["dvi", "reference"])
    ap.add_argument("--workload", default="7b")
    ap.add_argument("--extra", default="1b", help="second workload reported beside the headline ('' = none)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--layers", type=int, default=0, help="override the layer count (small profiling cases)")
    ap.add_argument("--prompt", type=int, default=0, help="override the prompt length (small profiling cases)")
    ap.add_argument("--no-megakernel", action="store_true",
                    help="run the draft phase one kernel per projection, attention and head (runtime option "
                         "megakernel = 0) instead of one persistent launch")
    ap.add_argument("--persistent", action="store_true",
                    help="run each layer's projections as one persistent launch (runtime option persistent = 1)")
    args = ap.parse_args()

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    w = workload(args.workload)
    if args.layers:
        from dataclasses import replace
        w = w.with_(shape=replace(w.shape, n_layers=args.layers), name=f"{w.name}-L{args.layers}")
    if args.prompt:
        w = w.with_(prompt_len=(args.prompt, args.prompt), name=f"{w.name}-p{args.prompt}")
    assert args.warmup >= 3, "at least 3 warm-up steps"

    if args.impl == "reference":
        return reference_arm(args, w, rank)

    import torch
    import torch.distributed as dist
    from paper_2510_05421_gb300 import DeviceWeights, update_config

    if world > 1:
        dist.init_process_group("gloo", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pk, pk_src = peaks()
    hbm = pk["hbm_gbs"]

    W = make_weights(w)
    dw = DeviceWeights.from_host(W, w.dtype, device=dev)
    P = make_prompts(w)
    U, K = w.update_every, w.k_spec
    gen_room = max(w.gen_tokens, (args.warmup + args.steps) * U * K)
    max_len = max(len(p) for p in P) + gen_room + 2 * K + 64
    eng = make_engine(w, dw, max_len, local, args.persistent, not args.no_megakernel)
    mk_ctas = eng.stats()["megakernel_ctas"]
    hyper = update_config(w.update)
    # prefill: sequence 0's prompt once to warm up, then every prompt timed
    # with CUDA events on the engine's stream (prompts already on the device)
    dP = [torch.from_numpy(p).to(dev) for p in P]
    eng.prefill(0, dP[0])
    pf0, pf1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    pf0.record(eng.stream)
    for b, p in enumerate(dP):
        eng.prefill(b, p)
    pf1.record(eng.stream)
    torch.cuda.synchronize(dev)
    pf_ms = pf0.elapsed_time(pf1)
    pf_tokens = sum(len(p) for p in P)
    chunk = eng.rt.max_prefill_chunk or (1024 if w.dtype == "bf16" else 128)
    pf_traffic = sum(prefill_bytes(w, len(p), chunk) for p in P)
    pf_alg = sum(prefill_alg_bytes(w, len(p)) for p in P)
    pf_flops = sum(prefill_flops(w, len(p)) for p in P)

    r = time_dvi(eng, w, hyper, args.warmup, args.steps, dev, world, clocks=True)
    ms_all, committed_all = combine_ranks(r["ms"], r["committed"], world)
    value = committed_all / (ms_all / 1e3)
    n_mid, draft_b, verify_b, d_ms, v_ms, u_ms = pass_rooflines(w, r, hbm)
    v_gbs = verify_b / (v_ms / 1e3) / 1e9
    d_gbs = draft_b / (d_ms / 1e3) / 1e9
    v_traffic = measured_traffic(w, n_mid, args.persistent)

    # greedy AR on the same engine, context and token count (rank-local)
    ar = time_ar(eng, dP, r["lens0"], r["committed"], dev)
    ar_ms_all, ar_tok_all = combine_ranks(ar["ms_per_step"] * ar["steps"], w.batch * ar["steps"], world)
    ar_value = ar_tok_all / (ar_ms_all / 1e3)

    e2e = None
    if not args.no_e2e:
        eng.close()
        eng = make_engine(w, dw, max(len(p) for p in P) + w.gen_tokens * K + 64, local, args.persistent,
                          not args.no_megakernel)
        eng.generate(P, 8, update_every=U, hyper=w.update, max_steps=2 * U)
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        toks, mats, h2d, d2h = eng.generate(P, w.gen_tokens, update_every=U, hyper=w.update)
        torch.cuda.synchronize(dev)
        dt = time.perf_counter() - t0
        nsteps = max(1, len(mats))
        ntok = sum(len(t) for t in toks)
        e2e = {"value": ntok / dt, "unit": "tokens/s", "h2d_bytes_per_step": h2d / nsteps,
               "d2h_bytes_per_step": d2h / nsteps,
               "note": (f"DVIEngine.generate(): {w.gen_tokens} tokens per sequence from pinned host prompts "
                        f"({len(P[0])} ids) to host token lists, prefill included, drafter updated every {U} "
                        f"steps; {len(mats)} decode steps, MAT {float(np.mean(mats)):.3f}")}
    eng.close()
    del eng, dw
    torch.cuda.empty_cache()

    extra = None
    if args.extra and not args.layers and not args.prompt:
        extra = extra_workload(args.extra, args, local, dev, pk)

    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_all / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
        "config": {"workload": w.name, "layers": w.shape.n_layers, "d_model": w.shape.d_model,
                   "batch": w.batch, "split_k": w.split_k, "k_spec": K, "prompt": len(P[0]),
                   "update_every": U, "lora_rank": w.lora_rank,
                   "step": f"{U} draft_verify_commit calls + 1 update_drafter",
                   "l2": "inputs larger than L2: ~13 GB of weights streamed per step",
                   "parallelism": "replicas" if world > 1 else "single GPU",
                   "projections": "persistent chain" if args.persistent else "one kernel each",
                   "draft_phase": (f"one persistent launch of {mk_ctas} CTAs (megakernel)" if mk_ctas
                                   else "one kernel per projection, attention and head")},
        "mean_accepted_length": r["mat"],
        "ar_tokens_per_s": ar_value,
        "speedup_vs_ar": value / ar_value,
        "ar": {"note": ("dvi_ar_step (greedy AR of the full model, CUDA-graph replay) on the same engine, "
                        "weights and starting context, timed over the same number of committed tokens"),
               "ms_per_step": ar["ms_per_step"], "steps": ar["steps"]},
        "prefill": {"tokens": pf_tokens, "ms": pf_ms, "tokens_per_s": pf_tokens / (pf_ms / 1e3), "chunk": chunk,
                    "roofline": prefill_roofline(pf_flops, pf_alg, pf_ms, pk, traffic=pf_traffic)},
        "roofline": {"bound": "hbm", "achieved": v_gbs, "peak": hbm, "unit": "GB/s", "frac": v_gbs / hbm,
                     "traffic": v_traffic, "kernel": "verify pass (layers k+1..L + LM head, CUDA-graph replay)",
                     "traffic_source": "profiles/verify_pass_dram_7b_width.md (ncu, 4-layer case scaled)"
                     if v_traffic else None,
                     "bytes_per_launch": verify_b, "ms_per_launch": v_ms, "peak_source": pk_src},
        "roofline_draft": {"bound": "hbm", "achieved": d_gbs, "peak": hbm, "unit": "GB/s", "frac": d_gbs / hbm,
                           "bytes_per_launch": draft_b, "ms_per_launch": d_ms},
        "update_ms": u_ms,
        "roofline_update": update_roofline(w, u_ms, hbm),
        "gpu_launches": r["launches"],
        "clocks": r["clocks"],
        "device_flags": r["status"],
    }
    if e2e:
        line["e2e"] = e2e
    if extra:
        line["extra_workload"] = extra
    if rank == 0 and world == 1 and not args.no_cpu:
        cores = os.cpu_count() or 1
        run = OracleRun(w, W)
        dvi = run.dvi(args.cpu_seconds)
        arc = run.ar(args.cpu_seconds / 2)
        line["cpu_baseline"] = cpu_baseline_dict(run, dvi, arc, cores)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())

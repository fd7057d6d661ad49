"""Benchmark of the batch-1 decoder forward pass on the Llama-3-8B shape.

One step = one request: reset, prefill of a 1024-token seeded prompt (TTFT),
then 256 greedy decode steps, all through the C ABI of libwici.so.  `value` is
decode tokens/s over the K timed steps (CUDA events on the library's stream;
weights and KV already in HBM); TTFT and achieved HBM bandwidth are reported
beside it.  The 16 GB of weights exceed L2 (129 MB) many times over, so no L2
flush is needed between steps.

Beside the decode roofline (`roofline`, the dominant kernel) the line carries
`prefill_roofline` (the request's prefill FLOPs / TTFT against the bf16 tensor
peak), `agentic`: the agentic long-context workload at the same shape
(4 turns of a 2048-token chunk plus 64 decode steps, 8448 cached), timed after
the K requests, with its four chunk prefills in aggregate against the bf16 peak,
`multi_tenant`: a 1B-shaped and the 8B-shaped model decoding at the same
time on SM shares of one GPU, per-tenant tokens/s, `q8`: the 8B request
with its per-layer matrices in the 8-bit block format, and `cnn_train`: the
paper's CNN-training sample (a 3x3 stride-2 convolution layer on 4 x 1024 x
224 x 224, forward and both gradients) against the bf16 tensor peak.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

--impl reference times the CPU oracle (numpy fp64) on a bounded sample of the
same workload: it is the baseline this path is compared with.  With N > 1 the
job runs as N independent replicas (one per GPU, launched by torchrun): the
decode path has no exchange step, so there is no collective.
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import gen  # noqa: E402

CFG = gen.LLAMA_8B
PROMPT = CFG.prompt_len        # 1024
DECODE = CFG.decode_steps      # 256
QUICK = False                  # profiling runs: no e2e, no per-kernel pass, no CPU baseline
METRIC = "bs=1 decode tok/s (Llama-3-8B shape, 1024-token prompt, 256 greedy steps)"
NOMINAL_HBM_GBS = 8000.0


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


KERNEL_SOURCES = ["paper_2608_24204_gb300/csrc/kernels_decode.cu", "paper_2608_24204_gb300/csrc/common.cuh",
                  "paper_2608_24204_gb300/csrc/plan.h"]


def decode_source_hash() -> str:
    import hashlib
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def profiled_traffic(profile: str):
    """DRAM bytes per launch recorded in a committed ncu summary, or None when the
    summary is missing or the decode kernel sources changed since the capture."""
    path = os.path.join(ROOT, "profiles", profile)
    try:
        with open(path) as f:
            text = f.read()
    except OSError:
        return None
    fields = {}
    for line in text.splitlines():
        line = line.strip().lstrip("-").strip()
        if ":" in line:
            k, v = line.split(":", 1)
            fields[k.strip()] = v.strip().strip("`")
    if fields.get("source_sha256") != decode_source_hash():
        return None
    try:
        return int(fields["traffic_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


class ClockSampler:
    """nvidia-smi clock/throttle samples every 200 ms while running."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        loaded = [s for s in sm if s > 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(smax), "samples": len(sm),
                "reasons": sorted(reasons)}


def max_over_ranks(values, world: int, device: str = "cuda"):
    """Element-wise maximum of `values` over all ranks (the slowest rank's times)."""
    import torch
    t = torch.tensor(list(values), dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t]


def job_tokens_per_s(world: int, local_tokens: int, slowest_s: float) -> float:
    """Whole-job decode rate: every replica decodes `local_tokens`; the job ends
    with the slowest one."""
    return world * local_tokens / slowest_s


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def cpu_oracle_sample(weights, budget_s: float = 20.0):
    """The oracle as it stands on the host cores: a 16-token prompt, then greedy
    decode steps until about `budget_s` of decode time (at least 1)."""
    import oracle
    m = oracle.OracleModel(CFG, weights, max_tokens=64)
    _, tok = m.prefill(gen.make_prompt(CFG, 16, seed=1))
    n, t0 = 0, time.perf_counter()
    while True:
        _, tok = m.decode(tok)
        n += 1
        if time.perf_counter() - t0 > budget_s or n >= 8:
            break
    dt = time.perf_counter() - t0
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    return {"value": n / dt, "unit": "tok/s", "cores": cores, "kind": "oracle",
            "sample": f"{CFG.name} weights, 16-token prompt, {n} greedy decode steps at context 17..{16 + n} "
                      f"(numpy fp64, {dt:.1f} s)"}


def measure_agentic(weights, WiciModel, torch, pk, runs: int = 3, cfg=None):
    """The agentic long-context workload at the 8B shape: 4 turns, each a
    2048-token chunk appended to the same cache (prefill) and then 64 greedy
    decode steps, ending at 8448 cached tokens.  Reported: the four chunk
    prefills in aggregate (the 8K-token prefill) against the bf16 tensor peak,
    and the decode steps against the HBM peak.  CUDA events on the library's
    stream; one untimed run first, then the median of `runs`."""
    cfg = cfg or gen.LLAMA_8B_AGENTIC
    T, steps, turns = cfg.prompt_len, cfg.decode_steps, cfg.turns
    model = WiciModel(cfg, max_tokens=turns * (T + steps), max_chunk=T).load(weights)
    prompts = [gen.make_prompt(cfg, T, seed=s) for s in cfg.prompt_seeds]
    st = model.stream
    pf_ms, dec_ms = [], []
    for r in range(runs + 1):
        model.reset()
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(turns)]
        for t in range(turns):
            ev[t][0].record(st)
            model.prefill(prompts[t])
            ev[t][1].record(st)
            model.decode(steps)
            ev[t][2].record(st)
        torch.cuda.synchronize()
        if r > 0:
            pf_ms.append([e[0].elapsed_time(e[1]) for e in ev])
            dec_ms.append([e[1].elapsed_time(e[2]) for e in ev])
    # the last turn's prefill kernels one by one (CUDA events around every launch)
    from paper_2608_24204_gb300 import wici
    model.reset()
    for t in range(turns - 1):
        model.prefill(prompts[t])
        model.decode(steps)
    prof = wici.wici_profile_prefill(model.ctx, prompts[turns - 1])
    model.close()
    P4 = (turns - 1) * (T + steps)
    attn_flops = cfg.n_layers * cfg.n_q_heads * cfg.head_dim * 4 * (T * P4 + T * (T + 1) // 2)
    n_a, ms_a = prof.get("prefill_attention", (0, float("nan")))
    attn_tf = attn_flops / (ms_a / 1000.0) / 1e12
    i = sorted(range(runs), key=lambda k: sum(pf_ms[k]))[runs // 2]
    pf, dec = pf_ms[i], dec_ms[i]
    flops = [gen.prefill_flops(cfg, T, t * (T + steps)) for t in range(turns)]
    tf = sum(flops) / (sum(pf) / 1000.0) / 1e12
    dec_bytes = sum(gen.decode_bytes_per_token(cfg, t * (T + steps) + T + j)
                    for t in range(turns) for j in range(1, steps + 1))
    dec_s = sum(dec) / 1000.0
    return {"workload": f"{cfg.name}: {turns} turns x ({T}-token chunk + {steps} greedy steps), "
                        f"{turns * (T + steps)} cached at the end",
            "prefill_ms": sum(pf), "prefill_ms_per_turn": pf, "prefill_flops": sum(flops),
            "prefill_roofline": {"bound": "tensor", "achieved": tf, "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
                                 "frac": tf / pk["bf16_tflops"],
                                 "frac_of_sustained": tf / pk["bf16_tflops_sustained"]},
            "last_turn_kernels_ms": {k: v[1] for k, v in prof.items()},
            "last_turn_attention": {"bound": "tensor", "launches": n_a, "ms": ms_a, "achieved": attn_tf,
                                    "peak": pk["bf16_tflops"], "unit": "TFLOP/s", "frac": attn_tf / pk["bf16_tflops"],
                                    "flops": attn_flops, "cached_before": P4, "chunk": T},
            "decode_tok_s": turns * steps / dec_s, "decode_gbs": dec_bytes / dec_s / 1e9,
            "decode_frac_of_8tbs": dec_bytes / dec_s / 1e9 / NOMINAL_HBM_GBS,
            "decode_frac_of_measured_hbm": dec_bytes / dec_s / 1e9 / pk["hbm_gbs"],
            "runs": runs}


def measure_q8(weights_8b, WiciModel, torch, pk, runs: int = 3):
    """The Llama-3-8B-shaped request with the seven per-layer matrices in the
    8-bit block format (int8 codes + one fp16 scale per 32; the embedding, norms
    and LM head stay bf16): 1024-token prompt, then 256 greedy decode steps.
    Decode tokens/s and bytes/s over the format's algorithmic bytes per token,
    the decode kernel's own launch time (CUDA events), and the TTFT."""
    from gen import q8 as gq
    from paper_2608_24204_gb300 import wici
    q8w = gq.make_q8_weights(CFG)
    model = WiciModel(CFG, max_tokens=PROMPT + DECODE + 16, max_chunk=PROMPT, q8=True).load(weights_8b, q8w)
    del q8w
    prompt = gen.make_prompt(CFG, PROMPT, seed=1)
    st = model.stream
    ttft, dec = [], []
    for r in range(runs + 1):
        model.reset()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        ev[0].record(st)
        model.prefill(prompt)
        ev[1].record(st)
        model.decode(DECODE)
        ev[2].record(st)
        torch.cuda.synchronize()
        if r > 0:
            ttft.append(ev[0].elapsed_time(ev[1]))
            dec.append(ev[1].elapsed_time(ev[2]))
    model.reset()
    model.prefill(prompt)
    n_prof = 8
    prof = wici.wici_profile_decode(model.ctx, n_prof)
    model.close()
    n_k, ms_k = prof["decode_step"]
    unit_bytes = sum(gen.decode_bytes_per_token(CFG, PROMPT + i, q8=True) for i in range(1, n_prof + 1)) / n_prof
    k_gbs = unit_bytes / (ms_k / n_k / 1000.0) / 1e9
    bytes_tok = sum(gen.decode_bytes_per_token(CFG, PROMPT + i, q8=True) for i in range(1, DECODE + 1)) / DECODE
    dec_s = statistics.median(dec) / 1000.0
    return {"workload": f"{CFG.name} in the 8-bit block format: prompt {PROMPT}, {DECODE} greedy decode steps",
            "decode_tok_s": DECODE / dec_s, "bytes_per_token": bytes_tok,
            "decode_gbs": bytes_tok * DECODE / dec_s / 1e9,
            "decode_frac_of_measured_hbm": bytes_tok * DECODE / dec_s / 1e9 / pk["hbm_gbs"],
            "decode_frac_of_8tbs": bytes_tok * DECODE / dec_s / 1e9 / NOMINAL_HBM_GBS,
            "roofline": {"bound": "hbm", "kernel": "decode_step (8-bit)", "achieved": k_gbs, "peak": pk["hbm_gbs"],
                         "unit": "GB/s", "frac": k_gbs / pk["hbm_gbs"], "bytes_per_launch": unit_bytes,
                         "avg_launch_us": ms_k / n_k * 1000.0},
            "ttft_ms": statistics.median(ttft), "runs": runs}


def measure_cnn_train(torch, pk, runs: int = 3):
    """The CNN-training sample (Sec. 5.4): one 3x3 stride-2 convolution layer on
    a 4 x 1024 x 224 x 224 input with 1024 output channels, forward plus the data
    and filter gradients, each timed with CUDA events (median of `runs` after one
    untimed run) against the bf16 tensor peak (each is 2 N P Q K C 9 FLOPs)."""
    from gen import conv as gc
    from paper_2608_24204_gb300 import wici
    s = gc.CNN_SAMPLE
    x, w, dy = gc.make_conv_inputs(s)
    dev = lambda a: torch.from_numpy(a.view(np.int16)).cuda()  # noqa: E731
    xd, wd, dyd = dev(x), dev(w), dev(dy)
    del x, w, dy
    shape = wici.wici_conv_shape(s.n, s.c, s.h, s.w, s.k)
    ws = torch.zeros(wici.wici_conv_workspace_bytes(shape), dtype=torch.uint8, device="cuda")
    y = torch.empty((s.n, s.p, s.q, s.k), device="cuda")
    dx = torch.empty((s.n, s.h, s.w, s.c), device="cuda")
    dw = torch.empty((s.k, 3, 3, s.c), device="cuda")
    st = torch.cuda.current_stream()
    calls = {"forward": lambda: wici.wici_conv_forward(st.cuda_stream, shape, xd.data_ptr(), wd.data_ptr(),
                                                       y.data_ptr(), ws.data_ptr()),
             "data_gradient": lambda: wici.wici_conv_backward_data(st.cuda_stream, shape, dyd.data_ptr(),
                                                                   wd.data_ptr(), dx.data_ptr(), ws.data_ptr()),
             "filter_gradient": lambda: wici.wici_conv_backward_filter(st.cuda_stream, shape, xd.data_ptr(),
                                                                       dyd.data_ptr(), dw.data_ptr(), ws.data_ptr())}
    ms = {k: [] for k in calls}
    for r in range(runs + 1):
        for k, f in calls.items():
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(st)
            f()
            e1.record(st)
            e1.synchronize()
            if r > 0:
                ms[k].append(e0.elapsed_time(e1))
    wici.wici_conv_status(st.cuda_stream, ws.data_ptr())
    fl = s.flops()
    out = {"workload": f"conv 3x3 stride 2 pad 1: x {s.n}x{s.c}x{s.h}x{s.w} (channels last, bf16), {s.k} filters; "
                       "forward, data gradient, filter gradient; fp32 outputs",
           "flops_each": fl, "peak": pk["bf16_tflops"], "unit": "TFLOP/s"}
    tot = 0.0
    for k in calls:
        m = statistics.median(ms[k])
        tot += m
        out[k] = {"ms": m, "tflops": fl / (m / 1000.0) / 1e12, "frac": fl / (m / 1000.0) / 1e12 / pk["bf16_tflops"]}
    out["step_ms"] = tot
    out["step_tflops"] = 3 * fl / (tot / 1000.0) / 1e12
    out["step_frac"] = out["step_tflops"] / pk["bf16_tflops"]
    return out


def measure_multi_tenant(weights_8b, WiciModel, torch, steps: int = 256):
    """Two tenants on one GPU, as in the paper's two-client microbenchmark: a
    Llama-3.2-1B-shaped model (512-token prompt) and the Llama-3-8B-shaped one
    (1024-token prompt), each with an SM share (a quarter and the rest) so that
    both persistent decode grids are resident at once, each on its own stream
    (the small model's at the higher priority).  Decode tokens/s of each
    tenant alone on its share, then with both decoding at the same time from
    two host threads; CUDA events on each tenant's stream."""
    import threading
    nsm = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    shares = {"small": nsm // 4, "large": nsm - nsm // 4}
    cfgs = {"small": gen.LLAMA_1B, "large": gen.LLAMA_8B}
    prompts = {k: gen.make_prompt(c, c.prompt_len, seed=1) for k, c in cfgs.items()}
    models = {}
    for k, c in cfgs.items():
        w = weights_8b if k == "large" else gen.make_weights(c)
        st = torch.cuda.Stream(priority=-1 if k == "small" else 0)
        models[k] = WiciModel(c, max_tokens=c.prompt_len + steps + 16, max_chunk=c.prompt_len, stream=st,
                              max_sms=shares[k]).load(w)

    def timed_decode(k, out):
        m = models[k]
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(m.stream)
        m.decode(steps)
        e1.record(m.stream)
        e1.synchronize()
        out[k] = steps / (e0.elapsed_time(e1) / 1000.0)

    def prime():
        for k, m in models.items():
            m.reset()
            m.prefill(prompts[k])
        torch.cuda.synchronize()

    prime()
    for k in models:               # warm-up (graph capture, row shares)
        timed_decode(k, {})
    alone = {}
    for k in models:
        prime()
        timed_decode(k, alone)
    prime()
    together = {}
    th = [threading.Thread(target=timed_decode, args=(k, together)) for k in models]
    for t in th:
        t.start()
    for t in th:
        t.join()
    for m in models.values():
        m.close()
    return {"workload": f"tenant small: {gen.LLAMA_1B.name} (prompt {gen.LLAMA_1B.prompt_len}), "
                        f"tenant large: {gen.LLAMA_8B.name} (prompt {gen.LLAMA_8B.prompt_len}); "
                        f"{steps} greedy decode steps each",
            "sm_share": shares, "stream_priority": {"small": -1, "large": 0},
            "tok_s_alone_on_share": alone, "tok_s_together": together,
            "unit": "tok/s"}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    t0 = time.time()
    weights = gen.make_weights(CFG)
    budget = max(5.0, 20.0 * args.steps / max(args.steps, 1))
    samples = []
    for _ in range(args.warmup + args.steps):
        samples.append(cpu_oracle_sample(weights, budget_s=budget / max(1, args.steps)))
    timed = samples[args.warmup:]
    val = statistics.median(s["value"] for s in timed)
    cb = dict(timed[-1])
    cb["value"] = val
    line = {"impl": "reference", "metric": METRIC, "value": val, "unit": "tok/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 / val,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded bf16 weights ~N(0,0.02), uniform-random prompt tokens)",
            "config": {"workload": f"{CFG.name}: prompt {PROMPT}, {DECODE} greedy decode steps (oracle sample)"},
            "cpu_baseline": cb,
            "e2e": {"value": val, "unit": "tok/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "wall_s": time.time() - t0}
    print(json.dumps(line), flush=True)
    return 0


def run_ours(args):
    global CFG, DECODE, QUICK
    if args.layers:
        CFG = CFG.with_(name=f"{CFG.name}-{args.layers}l", n_layers=args.layers)
    if args.decode_steps:
        DECODE = args.decode_steps
    QUICK = args.quick
    import torch
    from paper_2608_24204_gb300 import WiciModel, wici

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    dev = torch.cuda.current_device()
    pk = peaks()

    if QUICK and args.workload != "request":
        # profiling runs of the other measured workloads, at CFG's depth
        if args.workload == "agentic":
            cfg = gen.LLAMA_8B_AGENTIC.with_(n_layers=CFG.n_layers)
            out = measure_agentic(gen.make_weights(cfg), WiciModel, torch, pk, runs=args.steps, cfg=cfg)
        elif args.workload == "q8":
            out = measure_q8(gen.make_weights(CFG), WiciModel, torch, pk, runs=args.steps)
        else:
            out = measure_cnn_train(torch, pk, runs=args.steps)
        print(json.dumps({"profile_run": True, "workload": args.workload, **out}), flush=True)
        return 0

    t_setup = time.time()
    weights = gen.make_weights(CFG)
    max_tokens = PROMPT + DECODE + 16
    model = WiciModel(CFG, max_tokens=max_tokens, max_chunk=PROMPT).load(weights)
    prompt = gen.make_prompt(CFG, PROMPT, seed=1)
    stream = model.stream

    def one_request(ev=None):
        model.reset()
        if ev:
            ev[0].record(stream)
        model.prefill(prompt)
        if ev:
            ev[1].record(stream)
        model.decode(DECODE)
        if ev:
            ev[2].record(stream)

    for _ in range(args.warmup):
        one_request()
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    clocks = ClockSampler(dev)
    clocks.start()
    barrier()
    g0 = torch.cuda.Event(enable_timing=True)
    g1 = torch.cuda.Event(enable_timing=True)
    g0.record(stream)
    for k in range(args.steps):
        one_request(evs[k])
    g1.record(stream)
    barrier()
    clk = clocks.stop()
    total_ms = g0.elapsed_time(g1)
    ttft = [e[0].elapsed_time(e[1]) for e in evs]
    dec = [e[1].elapsed_time(e[2]) for e in evs]
    dec_s = sum(dec) / 1000.0
    local_tok = args.steps * DECODE
    dec_s_max, total_ms_max = max_over_ranks([dec_s, total_ms], world)
    value = job_tokens_per_s(world, local_tok, dec_s_max)

    # bytes per decoded token (weights + KV of the context), averaged over the 256 steps
    bytes_tok = sum(gen.decode_bytes_per_token(CFG, PROMPT + i) for i in range(1, DECODE + 1)) / DECODE
    step_gbs = bytes_tok * (local_tok / dec_s) / 1e9

    if QUICK:
        if rank == 0:
            print(json.dumps({"profile_run": True, "workload": CFG.name, "decode_steps": DECODE,
                              "value": value, "unit": "tok/s", "ttft_ms": statistics.median(ttft)}), flush=True)
        model.close()
        return 0

    # roofline of the dominant kernel, timed live with CUDA events on the library's stream
    model.reset()
    model.prefill(prompt)
    n_prof = 8
    prof = wici.wici_profile_decode(model.ctx, n_prof)
    if "decode_step" in prof:
        # the persistent decode kernel: one launch streams the whole step
        name = "decode_step"
        unit_bytes = sum(gen.decode_bytes_per_token(CFG, PROMPT + i) for i in range(1, n_prof + 1)) / n_prof
        traffic = profiled_traffic("decode_step_llama3-8b.md")
    else:
        # multi-launch decode (only for widths without a persistent instantiation;
        # not the case at this shape): the gate/up GEMV is the largest launch
        name = "gate_up_swiglu"
        H, F = CFG.hidden, CFG.ffn_dim
        unit_bytes = 2 * F * H * 2 + H * 2 + H * 4 + F * 4   # Wg|Wu + gain + x read + m written
        traffic = None
    n_k, ms_k = prof[name]
    k_gbs = unit_bytes / (ms_k / n_k / 1000.0) / 1e9
    roofline = {"bound": "hbm", "kernel": name, "achieved": k_gbs, "peak": pk["hbm_gbs"],
                "unit": "GB/s", "frac": k_gbs / pk["hbm_gbs"], "traffic": traffic,
                "peak_source": pk["source"], "bytes_per_launch": unit_bytes,
                "avg_launch_us": ms_k / n_k * 1000.0}
    kernel_share = {k: {"launches": v[0], "ms": v[1]} for k, v in prof.items()}

    # end to end through the public API: host prompt in pinned memory, one C-ABI call per token
    pinned = torch.from_numpy(prompt.copy()).pin_memory()
    host_prompt = pinned.numpy()
    e2e_steps = max(1, min(2, args.steps))
    e2e_dec, e2e_ttft = [], []
    for _ in range(e2e_steps):
        model.reset()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        tok = model.prefill(host_prompt)
        t1 = time.perf_counter()
        for _ in range(DECODE):
            tok = model.decode_step(-1)
        t2 = time.perf_counter()
        e2e_ttft.append((t1 - t0) * 1000)
        e2e_dec.append(t2 - t1)
    e2e_val = world * DECODE * e2e_steps / sum(e2e_dec)

    # prefill against the bf16 tensor peak: the request's TTFT covers the whole
    # 1024-token prefill (embed, 32 layers of GEMMs and attention, LM head)
    ttft_med = statistics.median(ttft)
    pf_flops = gen.prefill_flops(CFG, PROMPT)
    pf_tf = pf_flops / (ttft_med / 1000.0) / 1e12
    prefill_roofline = {"bound": "tensor", "achieved": pf_tf, "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
                        "frac": pf_tf / pk["bf16_tflops"], "frac_of_sustained": pf_tf / pk["bf16_tflops_sustained"],
                        "flops_per_prefill": pf_flops, "ttft_ms": ttft_med, "peak_source": pk["source"],
                        "what": f"algorithmic FLOPs of the {PROMPT}-token prefill / TTFT (CUDA events)"}

    agentic = tenants = q8 = cnn = None
    if not args.no_agentic and CFG.n_layers == gen.LLAMA_8B.n_layers:
        model.close()
        model = None
        agentic = measure_agentic(weights, WiciModel, torch, pk)
        tenants = measure_multi_tenant(weights, WiciModel, torch)
        q8 = measure_q8(weights, WiciModel, torch, pk)
        cnn = measure_cnn_train(torch, pk)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_oracle_sample(weights, budget_s=15.0)

    per_token = 1 if name == "decode_step" else 5 * CFG.n_layers + 1
    launches_per_step = (1 + CFG.n_layers * 7 + 1) + DECODE * per_token
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tok/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms_max / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded bf16 weights ~N(0,0.02), uniform-random prompt tokens)",
            "config": {"workload": f"{CFG.name}: L=32 H=4096 32q/8kv d=128 F=14336 V=128256; prompt {PROMPT}, "
                                   f"{DECODE} greedy decode steps per request",
                       "l2": "inputs larger than L2 (16 GB of weights streamed per token)",
                       "parallelism": "replicas" if world > 1 else "single GPU",
                       "accumulate": "fp32"},
            "ttft_ms": statistics.median(ttft),
            "decode_ms_per_token": dec_s / local_tok * 1000.0,
            "decode_gbs": step_gbs, "decode_frac_of_8tbs": step_gbs / (NOMINAL_HBM_GBS),
            "decode_frac_of_measured_hbm": step_gbs / pk["hbm_gbs"],
            "bytes_per_token": bytes_tok,
            "prefill_tflops": pf_tf,
            "roofline": roofline, "prefill_roofline": prefill_roofline, "agentic": agentic,
            "multi_tenant": tenants, "q8": q8, "cnn_train": cnn,
            "kernels": kernel_share, "cpu_baseline": cpu,
            "e2e": {"value": e2e_val, "unit": "tok/s", "h2d_bytes_per_step": PROMPT * 4,
                    "d2h_bytes_per_step": (DECODE + 1) * 4, "ttft_ms": statistics.median(e2e_ttft),
                    "how": "wici_prefill from pinned host tokens, then one wici_decode_step call per token, "
                           "wall clock"},
            "gpu_launches": launches_per_step * args.steps,
            "clocks": clk,
            "setup_s": time.time() - t_setup,
        }
        print(json.dumps(line), flush=True)
    if model is not None:
        model.close()
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-agentic", action="store_true",
                    help="skip the agentic, two-tenant, 8-bit-format and CNN measurements")
    ap.add_argument("--quick", action="store_true", help="profiling run: timed requests only")
    ap.add_argument("--decode-steps", type=int, default=0, help="profiling run: decode steps per request")
    ap.add_argument("--layers", type=int, default=0, help="profiling run: fewer layers (small ncu case)")
    ap.add_argument("--workload", default="request", choices=["request", "agentic", "q8", "cnn"],
                    help="profiling run (--quick): which measured workload to run")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())

"""Writes the full-size oracle records tests/golden/fullsize_<config>.npz from the
CPU oracle alone (no CUDA path is imported or run).

At the Llama-3-8B shape one oracle decode step streams the whole model through
numpy in fp64 (tens of seconds on a CPU), so the GPU tests cannot recompute
hundreds of full-depth steps on the fly.  This script runs them once:

  * llama3-8b: the 1024-token prompt (seed 1), then 64 decode steps;
  * llama3-8b-256: the same prompt, then all 256 decode steps of the request;
  * llama3-8b-agentic: 4 turns, each a 2048-token chunk (seeds 1..4) appended
    to the same cache and then 64 decode steps, ending at 8448 cached tokens;
  * llama3.2-1b: the 512-token prompt (seed 1), then all 128 decode steps of
    the configuration.

Decode steps are teacher-forced with a seeded token sequence (seed 101 + turn,
drawn like a prompt), so the oracle can take each turn's 64 steps as one causal
pass (`OracleModel.decode_forced`, pinned against step-by-step decode).  The GPU
test feeds the same tokens through `token_in` of wici_decode_step.

Per compared position (each turn's prefill, then every decode step) the file
keeps the oracle's greedy token and top-2 gap, its logits at 1024 fixed sample
indices and at its own 8 largest entries, and at a few positions (each turn's
prefill and last step, the first turn's first step) the whole logits vector.

Run (about half an hour on 8 cores):  python tests/golden/make_fullsize_golden.py [config ...]
"""
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import gen  # noqa: E402
import oracle  # noqa: E402

HERE = os.path.dirname(os.path.abspath(__file__))
N_SAMPLE = 1024
N_TOP = 8
FORCED_SEED0 = 101

WORKLOADS = {
    # name: (config, decode steps per turn)
    "llama3-8b": (gen.LLAMA_8B, 64),
    "llama3-8b-256": (gen.LLAMA_8B, 256),
    "llama3-8b-agentic": (gen.LLAMA_8B_AGENTIC, 64),
    "llama3.2-1b": (gen.LLAMA_1B, 128),
}


def sample_indices(vocab: int) -> np.ndarray:
    return np.sort(np.random.default_rng(20260).choice(vocab, N_SAMPLE, replace=False)).astype(np.int32)


def forced_tokens(cfg, turn: int, steps: int) -> np.ndarray:
    return gen.make_prompt(cfg, steps, seed=FORCED_SEED0 + turn)


def record(name: str, weights=None, log=print) -> str:
    cfg, steps = WORKLOADS[name]
    w = weights if weights is not None else gen.make_weights(cfg)
    turns = cfg.turns
    max_tokens = turns * (cfg.prompt_len + steps)
    ref = oracle.OracleModel(cfg, w, max_tokens=max_tokens, cache_bytes=0)
    idx = sample_indices(cfg.vocab)
    npos = 1 + steps
    tokens = np.zeros((turns, npos), np.int32)
    gaps = np.zeros((turns, npos), np.float64)
    sampled = np.zeros((turns, npos, N_SAMPLE), np.float32)
    top_idx = np.zeros((turns, npos, N_TOP), np.int32)
    top_val = np.zeros((turns, npos, N_TOP), np.float32)
    forced = np.zeros((turns, steps), np.int32)
    full_where, full = [], []
    keep_full = lambda t, p: p == 0 or p == npos - 1 or (t == 0 and p == 1)  # noqa: E731

    def store(t, p, logits):
        top = np.argsort(-logits, kind="stable")[:N_TOP]
        tokens[t, p] = oracle.greedy(logits)
        s = np.partition(logits, -2)[-2:]
        gaps[t, p] = float(s[1] - s[0])
        sampled[t, p] = logits[idx]
        top_idx[t, p] = top
        top_val[t, p] = logits[top]
        if keep_full(t, p):
            full_where.append((t, p))
            full.append(logits.astype(np.float32))

    for t in range(turns):
        prompt = gen.make_prompt(cfg, cfg.prompt_len, seed=cfg.prompt_seeds[t])
        t0 = time.time()
        logits, _ = ref.prefill(prompt)
        store(t, 0, logits)
        log(f"{name} turn {t}: prefill of {len(prompt)} at kv {ref.kv_len - len(prompt)} in {time.time() - t0:.0f} s")
        forced[t] = forced_tokens(cfg, t, steps)
        t0 = time.time()
        rows = ref.decode_forced(forced[t])
        for p in range(steps):
            store(t, 1 + p, rows[p])
        log(f"{name} turn {t}: {steps} forced decode steps in {time.time() - t0:.0f} s (kv {ref.kv_len})")
    path = os.path.join(HERE, f"fullsize_{name}.npz")
    np.savez_compressed(
        path, config=np.array(cfg.name), prompt_len=cfg.prompt_len, turns=turns, steps=steps,
        prompt_seeds=np.array(cfg.prompt_seeds[:turns], np.int32), forced=forced, sample_idx=idx,
        tokens=tokens, gaps=gaps, sampled=sampled, top_idx=top_idx, top_val=top_val,
        full_where=np.array(full_where, np.int32), full=np.stack(full))
    return path


if __name__ == "__main__":
    names = sys.argv[1:] or list(WORKLOADS)
    weights, key = None, None
    for n in names:
        cfg = WORKLOADS[n][0]
        if gen.tensor_specs(cfg) != key:          # the workloads share one set of weights
            t0 = time.time()
            weights, key = gen.make_weights(cfg), gen.tensor_specs(cfg)
            print(f"weights in {time.time() - t0:.0f} s", flush=True)
        print("wrote", record(n, weights, log=lambda m: print(m, flush=True)), flush=True)

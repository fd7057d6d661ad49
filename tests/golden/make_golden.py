"""Writes tests/golden/tiny_oracle.json from the CPU oracle alone (no CUDA path).

The file pins the oracle's output on the tiny configuration (2 layers, hidden
256, 4/2 heads, FFN 688, vocab 1024; prompt of 32 seeded tokens, 16 greedy
steps) so that any later change to the oracle's arithmetic shows up as a diff.
Run:  python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import gen  # noqa: E402
import oracle  # noqa: E402


def tiny_record():
    cfg = gen.TINY
    w = gen.make_weights(cfg)
    prompt = gen.make_prompt(cfg, cfg.prompt_len, seed=1)
    out = oracle.run_workload(cfg, w, [prompt], cfg.decode_steps)
    steps = []
    for logits, tok in out:
        top = np.argsort(-logits, kind="stable")[:5]
        steps.append({"token": int(tok),
                      "top5": [[int(i), float(logits[i])] for i in top],
                      "sum": float(logits.sum()), "sumsq": float((logits * logits).sum())})
    return {"config": cfg.name, "prompt_seed": 1, "prompt": [int(t) for t in prompt],
            "steps": steps}


if __name__ == "__main__":
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "tiny_oracle.json")
    with open(path, "w") as f:
        json.dump(tiny_record(), f, indent=1)
    print("wrote", path)

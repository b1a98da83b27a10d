"""Writes walk_stats.json: the work of the plain definition of C.mask() on each
decode workload, as bytes walked per (row, token) check.

The mask walk (Alg. 1 `mask`, Sec. 3.5 at lookahead k = infinity) checks each
token by stepping the automaton through its bytes until the end of the token or
the first byte that leaves the live states.  The number of such steps per check
is the algorithmic unit of work of a mask step (one transition lookup each); it
depends on where the sequences are, so it is averaged over the first decode
steps of the same seeded greedy trajectory the benchmark runs: rows start from
Workload.initial_configs(part=2), step i decodes logits(100 + i % n_buffers)
and every step is step_mask -> greedy argmax -> advance, all three taken from
the oracle.  Only the oracle and the seeded generators are used.

    python tests/golden/make_walk_stats.py [--steps 32] [--threads 8]
"""
from __future__ import annotations

import argparse
import json
import math
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
from paper_2403_06988_gb300 import synth  # noqa: E402

L2_BYTES = 129 * 1024 * 1024
OUT = os.path.join(HERE, "walk_stats.json")


def logit_buffers(w) -> int:
    """Number of rotating logits buffers the benchmark uses (more than twice the L2)."""
    esz = 2 if w.logits_dtype == "bf16" else 4
    return max(4, math.ceil(2.2 * L2_BYTES / (w.batch * w.vocab.n_tokens * esz)))


def trajectory_walk_steps(config: int, steps: int, threads: int):
    w = synth.workload(config)
    P = oracle.Problem.from_workload(w)
    stack = w.automaton.rules is not None
    states, stacks = w.initial_configs(part=2)
    nbuf = logit_buffers(w)
    checks = w.batch * w.vocab.n_tokens
    per_step = []
    for i in range(steps):
        sk = stacks if stack else None
        per_step.append(P.walk_steps(states, sk, n_threads=threads) / checks)
        mask, _, _ = P.step_mask(states, sk, n_threads=threads)
        arg, _, _ = oracle.mask_logits(w.logits(100 + i % nbuf), mask, want_logprobs=False, n_threads=threads)
        states, stacks, _ = P.advance(states, sk, arg, w.automaton.start)
        if not stack:
            stacks = None
    return w, per_step


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--steps", type=int, default=32)
    ap.add_argument("--threads", type=int, default=os.cpu_count() or 1)
    ap.add_argument("--configs", default="1,2,3,5")
    args = ap.parse_args()
    out = {}
    for c in [int(x) for x in args.configs.split(",")]:
        w, per = trajectory_walk_steps(c, args.steps, args.threads)
        out[w.name] = {"config": c, "batch": w.batch, "vocab": w.vocab.n_tokens, "steps": len(per),
                       "walk_steps_per_check_mean": sum(per) / len(per),
                       "walk_steps_per_check_last": per[-1], "walk_steps_per_check_step0": per[0]}
        print(w.name, out[w.name], flush=True)
    with open(OUT, "w") as f:
        json.dump(out, f, indent=1, sort_keys=True)
        f.write("\n")


if __name__ == "__main__":
    main()

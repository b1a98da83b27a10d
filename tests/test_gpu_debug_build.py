"""The debug build (libdomino_debug.so: every transition-table lookup checked
against the table's bounds, a violation reported in the device error word) run
on the workloads in a child process, whose binding loads it
(DOMINO_DEBUG_LIB=1): masks, next states and the decode step equal the
oracle's, and no check fires.  It stands in for a memory checker on the
table lookups, the walks' only data-dependent reads outside shared
memory's staged, validated records."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r'''
import os, sys
import numpy as np
import torch
sys.path.insert(0, ROOT); sys.path.insert(0, os.path.join(ROOT, "tests"))
from paper_2403_06988_gb300 import Domino, synth
from paper_2403_06988_gb300 import _binding as B
import oracle
from poison import assert_exact
assert B.LIB_PATH.endswith("libdomino_debug.so")
NT = os.cpu_count() or 1
def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()
for config, walk in ((3, "tree"), (3, "token"), (5, "token"), (2, "tree"), (1, "token")):
    os.environ["DOMINO_WALK"] = walk
    w = synth.workload(config)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    states, stacks = w.initial_configs()
    stack = w.automaton.rules is not None
    mask, nxt = d.step_mask(dev(states), dev(stacks.view(np.int64)) if stack else None, want_next=True)
    m_o, n_o, bad = oracle.Problem.from_workload(w).step_mask(states, stacks if stack else None, want_next=True,
                                                              n_threads=NT)
    assert bad == 0
    assert_exact(mask, m_o, "mask")
    assert_exact(nxt, n_o, "next")
    if w.logits_dtype == "bf16":
        lg = w.logits(0)
        lgt = dev(lg.view(np.int16)).view(torch.bfloat16)
        st = dev(states)
        sk = dev(stacks.view(np.int64)) if stack else None
        _, arg, _, _ = d.step_decode(st, sk, lgt, advance=True)
        arg_o, _, _ = oracle.mask_logits(lg, m_o, n_threads=NT)
        assert_exact(arg, np.asarray(arg_o, np.int32), "argmax")
    assert d.device_error() == 0, (config, walk, d.device_error())
    d.close()
w = synth.workload(2)
d = Domino.from_parts(w.automaton, w.vocab, device=0)
nxt, mask = d.precompute_table()
Q = w.automaton.n_states
m_o, n_o, _ = oracle.Problem.from_workload(w).step_mask(np.arange(Q, dtype=np.int32), want_next=True, n_threads=NT)
assert_exact(mask, m_o, "table mask")
assert_exact(nxt, n_o, "table next")
assert d.device_error() == 0
print("debug build ok")
'''


def test_debug_build_matches_oracle():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2403_06988_gb300 import build
    build.build(debug=True)
    env = dict(os.environ, DOMINO_DEBUG_LIB="1")
    r = subprocess.run([sys.executable, "-c", f"ROOT = {ROOT!r}\n" + CHILD], env=env, capture_output=True,
                       text=True, timeout=1200)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "debug build ok" in r.stdout

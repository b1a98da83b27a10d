"""The prefix-tree walk (Alg. 2's subterminal tree over byte classes, walked
once per row; selected here with DOMINO_WALK=tree, also for the automata whose
self-looping states make the per-token walk the default) against the oracle:
masks and next states bit-exact, on the workloads, the full state x token
table of config 2, tiny grammars with stacks and a ragged vocabulary.  Output
buffers start as 0xAB bytes (tests/poison.py)."""
import os

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

from paper_2403_06988_gb300 import Domino, synth  # noqa: E402
from paper_2403_06988_gb300 import _binding as B  # noqa: E402
import poison  # noqa: E402
from poison import assert_exact, assert_no_poison  # noqa: E402

TOL = 1e-3
NT = os.cpu_count() or 1


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2403_06988_gb300 import build
    build.build()


@pytest.fixture
def tree_walk(monkeypatch):
    monkeypatch.setenv("DOMINO_WALK", "tree")   # read when a handle is created


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


@pytest.mark.parametrize("config", [1, 2, 3, 5])
def test_tree_walk_step_mask(tree_walk, config):
    import oracle
    w = synth.workload(config)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    assert d.info()["walk_tree"] == 1
    states, stacks = w.initial_configs()
    has_stack = w.automaton.rules is not None
    mask, nxt = d.step_mask(dev(states), dev(stacks.view(np.int64)) if has_stack else None, want_next=True)
    P = oracle.Problem.from_workload(w)
    m_o, n_o, bad = P.step_mask(states, stacks if has_stack else None, want_next=True, n_threads=NT)
    assert bad == 0
    assert_exact(mask, m_o, "mask")
    assert_exact(nxt, n_o, "next")
    assert d.device_error() == 0
    d.close()


def test_tree_walk_precompute_config2(tree_walk):
    import oracle
    w = synth.workload(2)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    nxt, mask = d.precompute_table()
    Q = w.automaton.n_states
    m_o, n_o, _ = oracle.Problem.from_workload(w).step_mask(np.arange(Q, dtype=np.int32), want_next=True,
                                                             n_threads=NT)
    assert_exact(mask, m_o, "table mask")
    assert_exact(nxt, n_o, "table next")
    assert d.device_error() == 0
    d.close()


@pytest.mark.parametrize("n_tok,eos", [(1001, 0), (1003, 1002), (2050, 977), (4096, 4095)])
def test_tree_walk_precompute_ragged_vocab(tree_walk, n_tok, eos):
    """The precompute over 20000 states with vocabularies whose rows start off
    16-byte boundaries (V % 4 != 0); EOS first, last or inside a word (2000
    accepting states); with and without the mask."""
    import oracle
    w = synth.workload(4)
    a = w.automaton
    toks = [t for t in w.vocab.tokens()[:n_tok] if t][: n_tok - 1]
    toks.insert(eos, b"")
    v = synth.Vocab.from_tokens(toks, eos_id=eos)
    assert v.n_tokens == n_tok
    d = Domino.from_parts(a, v, device=0)
    assert d.info()["walk_tree"] == 1
    Q = a.n_states
    m_o, n_o, _ = oracle.Problem.from_parts(a, v).step_mask(np.arange(Q, dtype=np.int32), want_next=True,
                                                            n_threads=NT)
    assert m_o[:, eos >> 5].any() and (n_o[:, eos] != 0).any()
    nxt, mask = d.precompute_table()
    assert_exact(mask, m_o, "table mask")
    assert_exact(nxt, n_o, "table next")
    nxt, _ = d.precompute_table(want_mask=False)
    assert_exact(nxt, n_o, "table next without the mask")
    assert d.device_error() == 0
    d.close()


@pytest.mark.parametrize("name", ["dyck2", "int_regex", "dyck_ctx"])
def test_tree_walk_tiny_grammars(tree_walk, name):
    import oracle
    a = {"dyck2": lambda: synth.dyck2_pda(3), "int_regex": synth.int_regex_dfa,
         "dyck_ctx": lambda: synth.dyck_ctx_pda(3)}[name]()
    alpha = {"dyck2": b"{}[]a", "int_regex": b"-0123", "dyck_ctx": b"{}[]abc"}[name]
    v = synth.all_strings_vocab(alpha, 4)
    d = Domino.from_parts(a, v, device=0)
    assert d.info()["walk_tree"] == 1
    P = oracle.Problem.from_parts(a, v)
    states, stacks = [], []
    for q in range(1, a.n_states):
        for stk in ([], [0], [1], [1, 0], [0, 1, 1]):
            if len(stk) <= a.max_depth:
                states.append(q)
                stacks.append(synth.pack_stack(stk))
    states = np.array(states, np.int32)
    stacks = np.array(stacks, np.uint64)
    mask, nxt = d.step_mask(dev(states), dev(stacks.view(np.int64)), want_next=True)
    m_o, n_o, bad = P.step_mask(states, stacks, want_next=True)
    assert bad == 0
    assert_exact(mask, m_o, "mask")
    assert_exact(nxt, n_o, "next")
    d.close()


def test_tree_walk_long_chains(tree_walk):
    """Tokens of up to 700 bytes: runs of one-child nodes longer than one walk
    record (255 nodes), long shared prefixes that branch deep down, and
    tokens ending inside a run."""
    import oracle
    a = synth.int_regex_dfa()
    rng = np.random.default_rng(31)
    digits = np.frombuffer(b"0123456789", np.uint8)
    base = rng.choice(digits, 700).tobytes()
    toks = {base, base[:255], base[:256], base[:511], b"-" + base[:600], b"x" + base[:40]}
    for k in (3, 254, 255, 256, 300, 510, 699):   # branches deep inside the run
        toks.add(base[:k] + bytes([48 + (base[k] - 47) % 10]) + rng.choice(digits, 20).tobytes())
    while len(toks) < 400:
        toks.add(rng.choice(np.frombuffer(b"-0123456789x", np.uint8), int(rng.integers(1, 12))).tobytes())
    toks = sorted(toks)
    toks.insert(17, b"")   # EOS
    v = synth.Vocab.from_tokens(toks, eos_id=17)
    d = Domino.from_parts(a, v, device=0)
    assert d.info()["walk_tree"] == 1
    states = np.repeat(np.arange(a.n_states, dtype=np.int32), 3)
    mask, nxt = d.step_mask(dev(states), None, want_next=True)
    m_o, n_o, bad = oracle.Problem.from_parts(a, v).step_mask(states, want_next=True)
    assert bad == 0
    assert_exact(mask, m_o, "mask")
    assert_exact(nxt, n_o, "next")
    assert d.device_error() == 0
    d.close()

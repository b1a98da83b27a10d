"""The per-token walk (every token walked on its own from each row; the
kernel used when the vocabulary's prefix tree is not available, selected here
with DOMINO_WALK=token) against the oracle: masks and next states bit-exact,
the fused decode's argmax, lse and update as in test_gpu_step_decode.py.
Output buffers start as 0xAB bytes (tests/poison.py)."""
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
def token_walk(monkeypatch):
    monkeypatch.setenv("DOMINO_WALK", "token")   # read when a handle is created


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


@pytest.mark.parametrize("config", [1, 2, 3, 5])
def test_token_walk_step_mask(token_walk, config):
    import oracle
    w = synth.workload(config)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    assert d.info()["walk_tree"] == 0
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


def test_token_walk_precompute_config2(token_walk):
    import oracle
    w = synth.workload(2)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    nxt, mask = d.precompute_table()
    Q = w.automaton.n_states
    m_o, n_o, _ = oracle.Problem.from_workload(w).step_mask(np.arange(Q, dtype=np.int32), want_next=True,
                                                             n_threads=NT)
    assert_exact(mask, m_o, "table mask")
    assert_exact(nxt, n_o, "table next")
    d.close()


@pytest.mark.parametrize("config", [3, 5])
def test_token_walk_fused_step(token_walk, config):
    import oracle
    w = synth.workload(config)
    P = oracle.Problem.from_workload(w)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    states, stacks = w.initial_configs()
    has_stack = w.automaton.rules is not None
    lg = w.logits(13)
    t = dev(lg.view(np.int16))
    V, b = w.vocab.n_tokens, len(states)
    st = dev(states)
    sk = dev(stacks.view(np.int64)) if has_stack else None
    mask = poison.empty((b, d.info()["n_words"]), torch.int32)
    arg = poison.empty(b, torch.int32)
    lse = poison.empty(b, torch.float32)
    B.domino_step_decode(d.h, st, sk, b, t.data_ptr(), B.DTYPE_BF16, V, mask, arg, lse, None, st, sk)
    torch.cuda.synchronize()
    m_o, _, _ = P.step_mask(states, stacks if has_stack else None, n_threads=NT)
    a_o, l_o, _ = oracle.mask_logits(lg, m_o, n_threads=NT)
    s_o, k_o, _ = P.advance(states, stacks if has_stack else None, a_o, w.automaton.start)
    assert_exact(mask, m_o, "mask")
    assert_exact(arg, np.asarray(a_o, np.int32), "argmax")
    assert_no_poison(lse, "lse")
    fin = np.isfinite(l_o)
    assert np.abs(lse.cpu().numpy()[fin] - l_o[fin]).max(initial=0) < TOL
    assert_exact(st, s_o, "states")
    if has_stack:
        assert_exact(sk, k_o, "stacks")
    d.close()

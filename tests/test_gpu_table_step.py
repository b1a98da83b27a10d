"""Table-driven decode step (Sec. 3.5: masks computed before inference, looked
up while decoding) against the oracle's walk-based decode loop: argmax and
states bit-exact, lse and log-probs within 1e-3.  Output buffers start as 0xAB
bytes (tests/poison.py)."""
import functools
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


@functools.lru_cache(maxsize=None)
def workload(config):
    return synth.workload(config)


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def logits_tensor(x):
    return dev(x.view(np.int16)).view(torch.bfloat16) if x.dtype == np.uint16 else dev(x)


@pytest.mark.parametrize("config,steps,logprobs", [(1, 64, True), (2, 40, True), (3, 6, False)])
def test_table_driven_decode_loop_matches_oracle(config, steps, logprobs):
    import oracle
    w = workload(config)
    P = oracle.Problem.from_workload(w)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    nxt, tmask = d.precompute_table()
    states, _ = w.initial_configs()
    st = dev(states)
    s_o = states.copy()
    for i in range(steps):
        lg = w.logits(i)
        arg, lse, lp = d.mask_logits_table(logits_tensor(lg), tmask, st, want_logprobs=logprobs)
        d.advance_table(nxt, st, arg)
        m_o, _, _ = P.step_mask(s_o, None, n_threads=NT)
        a_o, l_o, lp_o = oracle.mask_logits(lg, m_o, want_logprobs=logprobs)
        s_o, _, _ = P.advance(s_o, None, a_o, w.automaton.start)
        assert_exact(arg, np.asarray(a_o, np.int32), f"argmax, step {i}")
        assert_no_poison(lse, f"lse, step {i}")
        lg_ = lse.cpu().numpy().astype(np.float64)
        fin = np.isfinite(l_o)
        assert (np.isfinite(lg_) == fin).all()
        assert np.abs(lg_[fin] - l_o[fin]).max(initial=0) < TOL
        if logprobs:
            assert_no_poison(lp, f"log-probs, step {i}")
            pg = lp.cpu().numpy().astype(np.float64)
            f2 = np.isfinite(lp_o)
            assert (np.isfinite(pg) == f2).all()
            assert np.abs(pg[f2] - lp_o[f2]).max(initial=0) < TOL
        assert (st.cpu().numpy() == s_o).all(), i
    assert d.device_error() == 0
    d.close()


def test_table_driven_invalid_states_and_tokens():
    w = workload(2)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    nxt, tmask = d.precompute_table()
    Q, V = w.automaton.n_states, w.vocab.n_tokens
    st = dev(np.array([-1, Q, 0, 1], np.int32))
    arg, lse, _ = d.mask_logits_table(logits_tensor(w.logits(0, batch=4)), tmask, st)
    a = arg.cpu().numpy()
    assert a[0] == -1 and a[1] == -1 and a[2] == -1     # out of range, out of range, dead state
    assert d.device_error() == B.DEVERR_BAD_STATE
    toks = dev(np.array([-1, V, w.vocab.eos_id, 5], np.int32))
    out = poison.empty(4, torch.int32)
    d.advance_table(nxt, dev(np.array([1, 1, 1, Q], np.int32)), toks, states_out=out)
    o = out.cpu().numpy()
    assert o[0] == w.automaton.start and o[1] == 0 and o[2] == w.automaton.start and o[3] == 0
    assert d.device_error() == B.DEVERR_BAD_TOKEN | B.DEVERR_BAD_STATE
    d.close()


def test_table_driven_refuses_pushdown():
    w = workload(5)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    x = torch.zeros(4, dtype=torch.int32, device="cuda")
    with pytest.raises(B.DominoError) as e:
        B.domino_advance_table(d.h, x, x, x, 1, x)
    assert e.value.status == -3
    with pytest.raises(B.DominoError) as e:
        B.domino_mask_logits_table(d.h, x, B.DTYPE_F32, 1, w.vocab.n_tokens, x, x, x)
    assert e.value.status == -3
    d.close()

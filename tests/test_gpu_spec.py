"""Count-based speculation (Sec. 3.6) through the C ABI against the oracle:
after the same sequence of count updates, the proposals, their number and the
configuration chains are identical; acceptance of a verification pass agrees.
Output buffers start as 0xAB bytes (tests/poison.py)."""
import functools
import os

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

from paper_2403_06988_gb300 import Domino, synth  # noqa: E402
from paper_2403_06988_gb300 import _binding as B  # noqa: E402
import poison  # noqa: E402
from poison import assert_exact  # noqa: E402

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


def host(t, dtype):
    return t.cpu().numpy().view(dtype)


class GpuSpec:
    def __init__(self, d, w):
        Q, V = w.automaton.n_states, w.vocab.n_tokens
        self.stack = w.automaton.rules is not None
        n_keys = Q * 3 if self.stack else Q
        self.d = d
        self.counts = torch.zeros((n_keys, V), dtype=torch.int32, device="cuda")
        self.best = torch.zeros(n_keys, dtype=torch.int64, device="cuda")
        self.reached = torch.zeros(n_keys, dtype=torch.int32, device="cuda")

    def update(self, states, stacks, tokens):
        B.domino_spec_update(self.d.h, self.counts, self.best, self.reached, dev(states),
                             dev(stacks.view(np.int64)) if stacks is not None else None, dev(tokens), len(states))

    def propose(self, states, stacks, s, permille):
        b = len(states)
        prop = poison.empty((b, s), torch.int32)
        n = poison.empty(b, torch.int32)
        cs = poison.empty((b, s + 1), torch.int32)
        ck = poison.empty((b, s + 1), torch.int64) if stacks is not None else None
        B.domino_spec_propose(self.d.h, self.best, self.reached, dev(states),
                              dev(stacks.view(np.int64)) if stacks is not None else None, b, s, permille, prop, n, cs,
                              ck)
        return prop, n, cs, ck


def trajectory(w, P, steps, batch):
    """The oracle's greedy decode: (states, stacks, tokens) of every step."""
    import oracle
    has_stack = w.automaton.rules is not None
    states, stacks = w.initial_configs(batch=batch)
    sk = stacks if has_stack else None
    out = []
    for i in range(steps):
        m, _, _ = P.step_mask(states, sk, n_threads=NT)
        arg, _, _ = oracle.mask_logits(w.logits(i % 7, batch=batch), m)   # logits repeat: choices recur
        out.append((states.copy(), None if sk is None else sk.copy(), arg.copy()))
        states, sk2, _ = P.advance(states, sk, arg, w.automaton.start)
        sk = sk2 if has_stack else None
    return out, states, sk


@pytest.mark.parametrize("config", [1, 2, 3, 5])
def test_proposals_match_oracle_after_the_same_updates(config):
    import oracle
    w = workload(config)
    P = oracle.Problem.from_workload(w)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    batch = min(w.batch, 64)
    traj, st_end, sk_end = trajectory(w, P, 16, batch)
    osp, gsp = oracle.Spec(P), GpuSpec(d, w)
    for st, sk, tok in traj:
        osp.update(st, sk, tok)
        gsp.update(st, sk, tok)
    probe = [(st_end, sk_end)] + [(st, sk) for st, sk, _ in traj[::5]]
    for states, stacks in probe:
        for s, permille in ((4, 0), (6, 400), (3, 900)):
            po, no, co, ko = osp.propose(states, stacks, s, permille)
            pg, ng, cg, kg = gsp.propose(states, stacks, s, permille)
            assert_exact(pg, po, "proposals")
            assert_exact(ng, no, "number of proposals")
            assert_exact(cg, co, "chain states")
            if ko is not None:
                assert_exact(kg, ko, "chain stacks")
    assert int(no.max()) >= 0
    d.close()


@pytest.mark.parametrize("config", [2, 5])
def test_accept_matches_oracle(config):
    import oracle
    w = workload(config)
    P = oracle.Problem.from_workload(w)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    batch, s = 32, 4
    traj, st_end, sk_end = trajectory(w, P, 12, batch)
    osp, gsp = oracle.Spec(P), GpuSpec(d, w)
    for st, sk, tok in traj:
        osp.update(st, sk, tok)
        gsp.update(st, sk, tok)
    prop, n, cs, ck = osp.propose(st_end, sk_end, s, 0)
    # verification pass: the constrained decode at every chain configuration
    flat_s = cs.reshape(-1)
    flat_k = ck.reshape(-1) if ck is not None else None
    m, _, _ = P.step_mask(flat_s, flat_k, n_threads=NT)
    lg = w.logits(3, batch=batch * (s + 1))
    dec, _, _ = oracle.mask_logits(lg, m)
    dec = dec.reshape(batch, s + 1)
    want = oracle.spec_accept(prop, n, dec)
    na = poison.empty(batch, torch.int32)
    tk = poison.empty(batch, torch.int32)
    so = poison.empty(batch, torch.int32)
    ko = poison.empty(batch, torch.int64) if ck is not None else None
    B.domino_spec_accept(d.h, dev(prop), dev(n), dev(dec), dev(cs), dev(ck.view(np.int64)) if ck is not None else None,
                         batch, s, na, tk, so, ko)
    assert_exact(na, np.asarray(want, np.int32), "accepted")
    k = host(na, np.int32)
    rows = np.arange(batch)
    assert_exact(tk, np.ascontiguousarray(dec[rows, k], np.int32), "next tokens")
    assert_exact(so, np.ascontiguousarray(cs[rows, k]), "chain states")
    if ck is not None:
        assert_exact(ko, np.ascontiguousarray(ck[rows, k]), "chain stacks")
    d.close()

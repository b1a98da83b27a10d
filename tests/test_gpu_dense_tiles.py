"""GPU parity on tiles whose rows are all live: the fullest walk-pair lists.

A tile of the step kernel holds up to 32 rows; each first class of the window
lists one walk pair per (token, group of up to four live rows).  When every
row survives every first byte, every class has eight groups, the rows of the
last group are 28..31 (the top of the 5-bit row fields), and the tile's list
reaches its bound of 1024 x 8 pairs.  For a pushdown automaton such a tile
also has more than four 32-pair chunks per warp, so its warps claim chunks
from a counter.  Batch 256 and 38 vocabulary windows make 8 x 38 = 304 tiles,
two per SM of a GB300, so the kernel takes 32 rows per tile.

Masks, next states, argmax and updated configurations: bit-exact against the
oracle; lse within 1e-3.  Outputs start as 0xAB bytes (tests/poison.py).
"""
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
ALPHA = b"abcdefghijklmnopqrstuvwxyz0123456789 .,:"
V = 38 * 1024 - 17          # 38 windows, the last one ragged
BATCH = 256


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2403_06988_gb300 import build
    build.build()


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def vocab(rng, extra=b""):
    """V - 1 distinct strings over ALPHA (+ extra), 1..12 bytes; about 3 % hold
    a byte no state accepts; EOS last."""
    toks = set()
    letters = np.frombuffer(ALPHA + extra, np.uint8)
    while len(toks) < V - 1:
        L = int(rng.integers(1, 13))
        t = bytearray(rng.choice(letters, L).tobytes())
        if rng.random() < 0.03:
            t[int(rng.integers(0, L))] = ord("#")
        toks.add(bytes(t))
    toks = sorted(toks)
    rng.shuffle(toks)
    return synth.Vocab.from_tokens(list(toks) + [b""], eos_id=V - 1)


def all_live_dfa():
    """Four accepting states; every byte of ALPHA leads from every state to a
    live state ((s + c) % 4 + 1), every other byte to the dead state."""
    delta = np.zeros((5, 256), np.int32)
    for s in range(1, 5):
        for c in ALPHA:
            delta[s][c] = (s + c) % 4 + 1
    live = np.array([0, 1, 1, 1, 1], np.uint8)
    return synth.Automaton(delta=delta, live=live, accepting=live.copy(), start=1, rules=None, max_depth=0,
                           name="all_live4")


def bracket_pda(max_depth=6):
    """One accepting scanner state looping on ALPHA, '{' / '[' push 0 / 1 and
    '}' / ']' pop them, depth <= max_depth."""
    b = synth._Builder()
    top = b.state("top", accepting=True)
    b.edge(top, ALPHA, top)
    b.push(top, b"{", 0, top)
    b.push(top, b"[", 1, top)
    b.pop(top, b"}", 0, (top, top, top))
    b.pop(top, b"]", 1, (top, top, top))
    return b.build(top, max_depth, "bracket_all_live")


def check_step(a, v, states, stacks, seed):
    import oracle
    d = Domino.from_parts(a, v, device=0)
    P = oracle.Problem.from_parts(a, v)
    has_stack = stacks is not None
    st = dev(states)
    sk = dev(stacks.view(np.int64)) if has_stack else None
    # the mask step with next states
    mask, nxt = d.step_mask(st, sk, want_next=True)
    m_o, n_o, bad = P.step_mask(states, stacks, want_next=True, n_threads=NT)
    assert bad == 0
    assert_exact(mask, m_o, "mask")
    assert_exact(nxt, n_o, "next")
    # the fused step: decode folded into the walk, rows advanced in place
    rng = np.random.default_rng(seed)
    lg = synth.f32_to_bf16_bits(rng.normal(0.0, 3.0, (len(states), V)).astype(np.float32))
    t = dev(lg.view(np.int16)).view(torch.bfloat16)
    m2 = poison.empty_like(mask)
    arg = poison.empty(len(states), torch.int32)
    lse = poison.empty(len(states), torch.float32)
    B.domino_step_decode(d.h, st, sk, len(states), t.data_ptr(), B.DTYPE_BF16, V, m2, arg, lse, None, st, sk)
    torch.cuda.synchronize()
    a_o, l_o, _ = oracle.mask_logits(lg, m_o, n_threads=NT)
    s_o, k_o, bad = P.advance(states, stacks, a_o, a.start)
    assert bad == 0
    assert_exact(m2, m_o, "mask of the fused step")
    assert_exact(arg, a_o, "argmax")
    assert_no_poison(lse, "lse")
    assert np.abs(lse.cpu().numpy().astype(np.float64) - l_o).max() < TOL
    assert (st.cpu().numpy() == s_o).all()
    if has_stack:
        assert (sk.cpu().numpy().view(np.uint64) == k_o).all()
    assert d.device_error() == 0
    d.close()
    return m_o


def test_all_rows_live_dfa():
    rng = np.random.default_rng(71)
    v = vocab(rng)
    a = all_live_dfa()
    states = rng.integers(1, 5, BATCH).astype(np.int32)
    m_o = check_step(a, v, states, None, 72)
    # nearly every token is allowed in every row: every class has 32 live rows
    assert np.unpackbits(m_o.view(np.uint8)).mean() > 0.9


def test_all_rows_live_pushdown_claims_chunks():
    rng = np.random.default_rng(81)
    v = vocab(rng, extra=b"{}[]")
    a = bracket_pda(6)
    states = np.full(BATCH, a.start, np.int32)
    stacks = np.array([synth.pack_stack(list(rng.integers(0, 2, int(rng.integers(0, 7)))))
                       for _ in range(BATCH)], np.uint64)
    m_o = check_step(a, v, states, stacks, 82)
    assert np.unpackbits(m_o.view(np.uint8)).mean() > 0.5

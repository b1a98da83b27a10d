"""ctypes wrapper around the plain-C oracle (oracle.c).

TEST INFRASTRUCTURE ONLY: imported by tests/, by __graft_entry__.smoke() and
by bench.py's CPU-baseline leg.  The product library never loads it.
Outputs are numpy arrays; lse and log-probs are float64.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "liboracle.so")
# A test may point the wrapper at another build of oracle.c (mutation tests).
_SO_OVERRIDE = os.environ.get("DOMINO_ORACLE_SO")

PUSH, POP = 1, 2
F32, BF16 = 0, 1


class Rule(ctypes.Structure):
    _fields_ = [("state", ctypes.c_int32), ("byte", ctypes.c_uint8), ("kind", ctypes.c_uint8),
                ("sym", ctypes.c_uint8), ("pad", ctypes.c_uint8), ("next_if_empty", ctypes.c_int32),
                ("next_if_top0", ctypes.c_int32), ("next_if_top1", ctypes.c_int32)]


def build(force: bool = False) -> str:
    """Compile liboracle.so with gcc (OpenMP over independent rows)."""
    src = os.path.join(_HERE, "oracle.c")
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= max(
            os.path.getmtime(src), os.path.getmtime(os.path.join(_HERE, "oracle.h"))):
        return _SO
    tmp = _SO + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-Wall", "-o", tmp, src, "-lm"],
                   check=True)
    os.replace(tmp, _SO)
    return _SO


_lib = None


def lib():
    global _lib
    if _lib is None:
        if _SO_OVERRIDE:
            L = ctypes.CDLL(_SO_OVERRIDE)
        else:
            build()
            L = ctypes.CDLL(_SO)
        P = ctypes.c_void_p
        L.oracle_new.restype = P
        L.oracle_new.argtypes = [P, P, ctypes.c_int32, ctypes.c_int32, P, ctypes.c_int32, P, P, P,
                                 ctypes.c_int32, ctypes.c_int32]
        L.oracle_free.argtypes = [P]
        L.oracle_check_token.restype = ctypes.c_int
        L.oracle_check_token.argtypes = [P, ctypes.c_int32, ctypes.c_uint64, ctypes.c_int32, P, P]
        L.oracle_step_mask.restype = ctypes.c_int64
        L.oracle_step_mask.argtypes = [P, P, P, ctypes.c_int32, P, P, ctypes.c_int32]
        L.oracle_mask_logits.restype = None
        L.oracle_mask_logits.argtypes = [P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, P, P,
                                         P, P, ctypes.c_int32]
        L.oracle_walk_steps.restype = ctypes.c_int64
        L.oracle_walk_steps.argtypes = [P, P, P, ctypes.c_int32, ctypes.c_int32]
        L.oracle_philox4x32_10.restype = None
        L.oracle_philox4x32_10.argtypes = [P, ctypes.c_uint32, ctypes.c_uint32]
        L.oracle_ln_f32.restype = ctypes.c_float
        L.oracle_ln_f32.argtypes = [ctypes.c_float]
        L.oracle_mask_sample.restype = None
        L.oracle_mask_sample.argtypes = [P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, P,
                                         ctypes.c_float, ctypes.c_uint64, ctypes.c_uint64, P, ctypes.c_int32]
        L.oracle_spec_new.restype = P
        L.oracle_spec_new.argtypes = [P]
        L.oracle_spec_free.argtypes = [P]
        L.oracle_spec_update.restype = None
        L.oracle_spec_update.argtypes = [P, P, P, P, ctypes.c_int32]
        L.oracle_spec_propose.restype = None
        L.oracle_spec_propose.argtypes = [P, P, P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, P, P, P, P]
        L.oracle_spec_accept.restype = None
        L.oracle_spec_accept.argtypes = [P, P, P, ctypes.c_int32, ctypes.c_int32, P]
        L.oracle_advance.restype = ctypes.c_int64
        L.oracle_advance.argtypes = [P, P, P, P, ctypes.c_int32, ctypes.c_int32, P, P]
        _lib = L
    return _lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def rules_array(rules) -> Tuple[Optional[ctypes.Array], int]:
    """numpy structured rule records -> ctypes array of Rule."""
    if rules is None or len(rules) == 0:
        return None, 0
    arr = (Rule * len(rules))()
    for i, r in enumerate(rules):
        arr[i] = Rule(int(r["state"]), int(r["byte"]), int(r["kind"]), int(r["sym"]), 0,
                      int(r["next_if_empty"]), int(r["next_if_top0"]), int(r["next_if_top1"]))
    return arr, len(rules)


class Problem:
    """A vocabulary plus a scanner table (and optional bracket rules)."""

    def __init__(self, data, offsets, eos_id, delta, live, accepting=None, rules=None, max_depth=0):
        self.V = int(len(offsets) - 1)
        self.W = (self.V + 31) // 32
        self.eos_id = int(eos_id)
        self.n_states = int(delta.shape[0])
        self._keep = [np.ascontiguousarray(data, dtype=np.uint8), np.ascontiguousarray(offsets, dtype=np.int64),
                      np.ascontiguousarray(delta, dtype=np.int32), np.ascontiguousarray(live, dtype=np.uint8),
                      None if accepting is None else np.ascontiguousarray(accepting, dtype=np.uint8)]
        rarr, nr = rules_array(rules)
        self._rules = rarr
        d, o, dl, lv, ac = self._keep
        h = lib().oracle_new(_ptr(d), _ptr(o), self.V, self.eos_id, _ptr(dl), self.n_states, _ptr(lv), _ptr(ac),
                             ctypes.cast(rarr, ctypes.c_void_p) if rarr is not None else None, nr, int(max_depth))
        if not h:
            raise ValueError("oracle rejected the problem")
        self._h = h

    @staticmethod
    def from_workload(w) -> "Problem":
        a, v = w.automaton, w.vocab
        return Problem(v.data, v.offsets, v.eos_id, a.delta, a.live, a.accepting, a.rules, a.max_depth)

    @staticmethod
    def from_parts(automaton, vocab) -> "Problem":
        a, v = automaton, vocab
        return Problem(v.data, v.offsets, v.eos_id, a.delta, a.live, a.accepting, a.rules, a.max_depth)

    def __del__(self):
        h = getattr(self, "_h", None)
        if h and _lib is not None:
            _lib.oracle_free(h)
            self._h = None

    def check(self, state: int, stack: int, token: int) -> Tuple[int, int, int]:
        """(status, next_state, next_stack); status 1 allowed, 0 rejected, -1 invalid."""
        ns = ctypes.c_int32(0)
        nw = ctypes.c_uint64(0)
        r = lib().oracle_check_token(self._h, int(state), int(stack) & 0xFFFFFFFFFFFFFFFF, int(token),
                                     ctypes.byref(ns), ctypes.byref(nw))
        return r, ns.value, nw.value

    def step_mask(self, states, stacks=None, want_next=False, n_threads=1):
        states = np.ascontiguousarray(states, dtype=np.int32)
        B = states.shape[0]
        stacks = None if stacks is None else np.ascontiguousarray(stacks, dtype=np.uint64)
        mask = np.zeros((B, self.W), dtype=np.uint32)
        nxt = np.zeros((B, self.V), dtype=np.int32) if want_next else None
        bad = lib().oracle_step_mask(self._h, _ptr(states), _ptr(stacks), B, _ptr(mask), _ptr(nxt), int(n_threads))
        return mask, nxt, int(bad)

    def walk_steps(self, states, stacks=None, n_threads=1) -> int:
        """Bytes the plain definition walks to check every token from every row."""
        states = np.ascontiguousarray(states, dtype=np.int32)
        stacks = None if stacks is None else np.ascontiguousarray(stacks, dtype=np.uint64)
        return int(lib().oracle_walk_steps(self._h, _ptr(states), _ptr(stacks), states.shape[0], int(n_threads)))

    def advance(self, states, stacks, tokens, start_state):
        states = np.ascontiguousarray(states, dtype=np.int32)
        B = states.shape[0]
        stacks = None if stacks is None else np.ascontiguousarray(stacks, dtype=np.uint64)
        tokens = np.ascontiguousarray(tokens, dtype=np.int32)
        so = np.zeros(B, dtype=np.int32)
        wo = np.zeros(B, dtype=np.uint64)
        bad = lib().oracle_advance(self._h, _ptr(states), _ptr(stacks), _ptr(tokens), B, int(start_state),
                                   _ptr(so), _ptr(wo))
        return so, wo, int(bad)


class Spec:
    """Count-based speculative proposals (Sec. 3.6) over a Problem's automaton."""

    def __init__(self, problem: "Problem"):
        self.problem = problem                    # keeps the automaton alive
        self._h = lib().oracle_spec_new(problem._h)

    def __del__(self):
        h = getattr(self, "_h", None)
        if h and _lib is not None:
            _lib.oracle_spec_free(h)
            self._h = None

    def update(self, states, stacks, tokens) -> None:
        states = np.ascontiguousarray(states, dtype=np.int32)
        stacks = None if stacks is None else np.ascontiguousarray(stacks, dtype=np.uint64)
        tokens = np.ascontiguousarray(tokens, dtype=np.int32)
        lib().oracle_spec_update(self._h, _ptr(states), _ptr(stacks), _ptr(tokens), states.shape[0])

    def propose(self, states, stacks, s: int, min_permille: int):
        """(proposals [B][s], n_prop [B], chain_states [B][s+1], chain_stacks [B][s+1] or None)."""
        states = np.ascontiguousarray(states, dtype=np.int32)
        B = states.shape[0]
        stacks = None if stacks is None else np.ascontiguousarray(stacks, dtype=np.uint64)
        prop = np.zeros((B, s), np.int32)
        n = np.zeros(B, np.int32)
        cs = np.zeros((B, s + 1), np.int32)
        ck = np.zeros((B, s + 1), np.uint64) if stacks is not None else None
        lib().oracle_spec_propose(self._h, _ptr(states), _ptr(stacks), B, int(s), int(min_permille), _ptr(prop),
                                  _ptr(n), _ptr(cs), _ptr(ck))
        return prop, n, cs, ck


def spec_accept(proposals, n_prop, decoded) -> np.ndarray:
    proposals = np.ascontiguousarray(proposals, dtype=np.int32)
    n_prop = np.ascontiguousarray(n_prop, dtype=np.int32)
    decoded = np.ascontiguousarray(decoded, dtype=np.int32)
    B, s = proposals.shape
    out = np.zeros(B, np.int32)
    lib().oracle_spec_accept(_ptr(proposals), _ptr(n_prop), _ptr(decoded), B, s, _ptr(out))
    return out


def mask_logits(logits: np.ndarray, mask: np.ndarray, n_tokens: Optional[int] = None, want_lse=True,
                want_logprobs=False, n_threads=1):
    """logits: float32 [B][>=V] or uint16 bf16 bits [B][>=V] (row stride = shape[1])."""
    logits = np.ascontiguousarray(logits)
    dtype = BF16 if logits.dtype == np.uint16 else F32
    if dtype == F32:
        logits = logits.astype(np.float32, copy=False)
    B, stride = logits.shape
    V = stride if n_tokens is None else int(n_tokens)
    mask = np.ascontiguousarray(mask, dtype=np.uint32)
    arg = np.zeros(B, dtype=np.int32)
    lse = np.zeros(B, dtype=np.float64) if want_lse else None
    lp = np.zeros((B, V), dtype=np.float64) if want_logprobs else None
    lib().oracle_mask_logits(_ptr(logits), dtype, B, V, stride, _ptr(mask), _ptr(arg), _ptr(lse), _ptr(lp),
                             int(n_threads))
    return arg, lse, lp


def philox4x32_10(ctr, key0: int, key1: int) -> np.ndarray:
    """Philox4x32-10 of one 4-word counter."""
    c = np.ascontiguousarray(np.asarray(ctr, dtype=np.uint32).copy())
    lib().oracle_philox4x32_10(_ptr(c), int(key0) & 0xFFFFFFFF, int(key1) & 0xFFFFFFFF)
    return c


def ln_f32(x: float) -> float:
    return float(lib().oracle_ln_f32(float(x)))


def mask_sample(logits: np.ndarray, mask: np.ndarray, temperature: float, seed: int, offset: int,
                n_tokens: Optional[int] = None, n_threads: int = 1) -> np.ndarray:
    """Gumbel-max draw per row over the allowed tokens (tokens int32 [batch], -1 when none)."""
    batch = logits.shape[0]
    V = logits.shape[1] if n_tokens is None else n_tokens
    dtype = BF16 if logits.dtype == np.uint16 else F32
    lg = np.ascontiguousarray(logits)
    mask = np.ascontiguousarray(mask, dtype=np.uint32)
    out = np.zeros(batch, dtype=np.int32)
    lib().oracle_mask_sample(_ptr(lg), dtype, batch, V, lg.shape[1], _ptr(mask), float(temperature),
                             int(seed) & 0xFFFFFFFFFFFFFFFF, int(offset) & 0xFFFFFFFFFFFFFFFF, _ptr(out),
                             int(n_threads))
    return out


def bits_of(mask_row: np.ndarray, n_tokens: int) -> np.ndarray:
    """Unpack one mask row to a bool vector of length n_tokens."""
    b = np.unpackbits(mask_row.astype("<u4").view(np.uint8), bitorder="little")
    return b[:n_tokens].astype(bool)

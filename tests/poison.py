"""Poison-filled output buffers for the GPU parity tests.

Every output buffer a GPU test hands to the library is filled with 0xAB bytes
before the call, so that a word a kernel never writes keeps that pattern
instead of whatever the allocator returned (often zero, which is also the
right value for most words of a sparse mask).

- Outputs compared exactly with the oracle: equality proves every word was
  written, provided the oracle's own value is not the pattern.
  `assert_exact` checks both.
- Outputs compared within a tolerance (lse, log-probs): `assert_no_poison`
  checks that no 32-bit word still holds 0xABABABAB. As an fp32 value that is
  -1.2e-12, which a tolerance of 1e-3 around 0 would let through.
"""
import numpy as np

POISON_BYTE = 0xAB
POISON_U32 = 0xABABABAB
POISON_U64 = 0xABABABABABABABAB


def empty(shape, dtype, device="cuda", pin=False):
    import torch
    if pin:
        t = torch.empty(shape, dtype=dtype).pin_memory()
    else:
        t = torch.empty(shape, dtype=dtype, device=device)
    if t.numel():
        t.view(torch.uint8).fill_(POISON_BYTE)
    return t


def empty_like(t):
    return empty(tuple(t.shape), t.dtype, t.device)


def host(shape, dtype):
    """A numpy output buffer filled with the pattern."""
    a = np.empty(shape, dtype)
    a.view(np.uint8).fill(POISON_BYTE)
    return a


def _np(x):
    if hasattr(x, "detach"):
        x = x.detach().cpu().numpy()
    return np.ascontiguousarray(x)


def _words(a):
    a = _np(a)
    if a.dtype.itemsize == 8:
        return a.view(np.uint64), POISON_U64
    if a.dtype.itemsize == 4:
        return a.view(np.uint32), POISON_U32
    raise TypeError(f"no poison word for {a.dtype}")


def assert_no_poison(out, what=""):
    w, p = _words(out)
    bad = np.flatnonzero(w.reshape(-1) == p)
    assert bad.size == 0, f"{what}: {bad.size} words left unwritten (first at flat index {bad[0]})"


def assert_exact(out, expected, what=""):
    """out == expected word for word (pad bits included), and the expected
    value holds no poison word, so that equality proves every word was
    written."""
    o = _np(out)
    e = np.ascontiguousarray(expected)
    ow, _ = _words(o)
    ew, p = _words(e)
    assert ow.shape == ew.shape, f"{what}: shape {ow.shape} != {ew.shape}"
    assert not (ew == p).any(), f"{what}: the expected value holds the poison pattern"
    neq = np.flatnonzero(ow.reshape(-1) != ew.reshape(-1))
    assert neq.size == 0, (f"{what}: {neq.size} words differ; first at flat index {neq[0]}: "
                           f"{int(ow.reshape(-1)[neq[0]]):#x} != {int(ew.reshape(-1)[neq[0]]):#x}")

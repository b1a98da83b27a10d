"""ctypes binding of libdomino.so (include/domino.h).

Argument marshalling only: every function here has the name of the C entry
point it calls, turns torch tensors / numpy arrays into pointers and the
current CUDA stream into a cudaStream_t, and raises DominoError on a non-zero
status.  All computation happens in the library's kernels.  Importing this
module fails loudly when libdomino.so has not been built.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
# DOMINO_DEBUG_LIB=1: the bounds-checked build (build.build(debug=True))
LIB_PATH = os.path.join(_PKG, "libdomino_debug.so" if os.environ.get("DOMINO_DEBUG_LIB") == "1" else "libdomino.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "domino.h")

DOMINO_OK = 0
DTYPE_F32 = 0
DTYPE_BF16 = 1
DEVERR_BAD_STATE = 1
DEVERR_BAD_STACK = 2
DEVERR_BAD_TOKEN = 4
DEVERR_INTERNAL = 8
STATUS = {0: "OK", -1: "E_INVALID_ARG", -2: "E_NOT_LOADED", -3: "E_UNSUPPORTED", -4: "E_OOM", -5: "E_CUDA",
          -6: "E_NO_DEVICE"}


class DominoError(RuntimeError):
    def __init__(self, fn: str, status: int, text: str):
        super().__init__(f"{fn} failed: {STATUS.get(status, status)} ({text})")
        self.status = status


class StackRule(ctypes.Structure):
    _fields_ = [("state", ctypes.c_int32), ("byte", ctypes.c_uint8), ("kind", ctypes.c_uint8),
                ("sym", ctypes.c_uint8), ("pad", ctypes.c_uint8), ("next_if_empty", ctypes.c_int32),
                ("next_if_top0", ctypes.c_int32), ("next_if_top1", ctypes.c_int32)]


class Info(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "n_tokens", "n_words", "eos_id", "max_token_len", "n_states", "n_classes", "start_state", "max_depth",
        "n_rules", "has_stack", "table_in_smem", "device")] + [("device_bytes", ctypes.c_int64), ("walk_tree", ctypes.c_int32),
                                                              ("tree_units", ctypes.c_int32)]


_lib = None
P = ctypes.c_void_p
I32 = ctypes.c_int32
I64 = ctypes.c_int64

_SIGS = {
    "domino_create": [P, I32],
    "domino_destroy": [P],
    "domino_load_vocab": [P, P, P, I32, I32],
    "domino_load_automaton": [P, P, I32, P, P, I32, P, I32, I32],
    "domino_get_info": [P, P],
    "domino_get_byte_classes": [P, P],
    "domino_get_prefix_tree": [P, P, I64, P, I64, P, I64, P, I64, P],
    "domino_precompute_table": [P, P, P, P],
    "domino_step_mask": [P, P, P, I32, P, P, P],
    "domino_mask_logits": [P, P, I32, I32, I64, P, P, P, P, P],
    "domino_advance": [P, P, P, P, I32, P, P, P],
    "domino_decode_step_host": [P, P, I32, I32, P, P, P, P, P],
    "domino_get_device_error": [P, P, P],
    "domino_mask_logits_noalloc": [P, I32, I32, I32, I64, P, P, P, P, P],
    "domino_mask_logits_table": [P, P, I32, I32, I64, P, P, P, P, P, P],
    "domino_advance_table": [P, P, P, P, I32, P, P],
    "domino_mask_sample": [P, P, I32, I32, I64, P, ctypes.c_float, ctypes.c_uint64, ctypes.c_uint64, P, P],
    "domino_opportunistic_step": [P, P, I32, I32, I64, P, P, P, P, P, P],
    "domino_spec_update": [P, P, P, P, P, P, P, I32, P],
    "domino_spec_propose": [P, P, P, P, P, I32, I32, I32, P, P, P, P, P],
    "domino_spec_accept": [P, P, P, P, P, P, I32, I32, P, P, P, P, P],
    "domino_step_decode": [P, P, P, I32, P, I32, I64, P, P, P, P, P, P, P],
}


def lib() -> ctypes.CDLL:
    """Loads libdomino.so; raises when it has not been built (no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{os.path.basename(LIB_PATH)} is not built ({LIB_PATH}); run "
                              "__graft_entry__.build() or python -m paper_2403_06988_gb300.build "
                              "(build.build(debug=True) for the debug library)")
        L = ctypes.CDLL(LIB_PATH)
        for name, args in _SIGS.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = ctypes.c_int
        L.domino_status_string.argtypes = [ctypes.c_int]
        L.domino_status_string.restype = ctypes.c_char_p
        _lib = L
    return _lib


def header_symbols():
    """Entry points declared in include/domino.h."""
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:int|const char\*)\s+(domino_\w+)\s*\(", text, flags=re.M)))


def _check(fn: str, status: int):
    if status != DOMINO_OK:
        raise DominoError(fn, status, lib().domino_status_string(status).decode())


def _ptr(x) -> Optional[int]:
    """Device or host address of a torch tensor / numpy array (None passes NULL)."""
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        assert x.flags["C_CONTIGUOUS"]
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        assert x.is_contiguous()
        return x.data_ptr()
    if isinstance(x, int):
        return x
    raise TypeError(type(x))


def _stream(stream) -> Optional[int]:
    if stream is not None:
        return stream if isinstance(stream, int) else stream.cuda_stream
    import torch
    return torch.cuda.current_stream().cuda_stream


def status_string(status: int) -> str:
    return lib().domino_status_string(int(status)).decode()


# ----------------------------------------------------------------------------
# one function per entry point
# ----------------------------------------------------------------------------
def domino_create(cuda_device: int) -> int:
    h = ctypes.c_void_p()
    _check("domino_create", lib().domino_create(ctypes.byref(h), int(cuda_device)))
    return h.value


def domino_destroy(h: int) -> None:
    _check("domino_destroy", lib().domino_destroy(h))


def domino_load_vocab(h: int, data: np.ndarray, offsets: np.ndarray, n_tokens: int, eos_id: int) -> None:
    data = np.ascontiguousarray(data, dtype=np.uint8)
    offsets = np.ascontiguousarray(offsets, dtype=np.int64)
    _check("domino_load_vocab", lib().domino_load_vocab(h, _ptr(data), _ptr(offsets), int(n_tokens), int(eos_id)))


def rules_to_ctypes(rules):
    if rules is None or len(rules) == 0:
        return None, 0
    arr = (StackRule * len(rules))()
    for i, r in enumerate(rules):
        arr[i] = StackRule(int(r["state"]), int(r["byte"]), int(r["kind"]), int(r["sym"]), int(r["pad"]),
                           int(r["next_if_empty"]), int(r["next_if_top0"]), int(r["next_if_top1"]))
    return arr, len(rules)


def domino_load_automaton(h: int, delta: np.ndarray, n_states: int, live: np.ndarray, accepting, start_state: int,
                          rules, n_rules: Optional[int], max_depth: int) -> None:
    delta = np.ascontiguousarray(delta, dtype=np.int32)
    live = np.ascontiguousarray(live, dtype=np.uint8)
    acc = None if accepting is None else np.ascontiguousarray(accepting, dtype=np.uint8)
    if isinstance(rules, ctypes.Array):
        arr, n = rules, len(rules)
    else:
        arr, n = rules_to_ctypes(rules)
    if n_rules is not None:
        n = int(n_rules)
    _check("domino_load_automaton", lib().domino_load_automaton(
        h, _ptr(delta), int(n_states), _ptr(live), _ptr(acc), int(start_state),
        ctypes.cast(arr, ctypes.c_void_p) if arr is not None else None, n, int(max_depth)))


def domino_get_info(h: int) -> dict:
    info = Info()
    _check("domino_get_info", lib().domino_get_info(h, ctypes.byref(info)))
    return {name: getattr(info, name) for name, _ in Info._fields_}


def domino_get_byte_classes(h: int) -> np.ndarray:
    out = np.zeros(256, dtype=np.uint8)
    _check("domino_get_byte_classes", lib().domino_get_byte_classes(h, _ptr(out)))
    return out


def domino_get_prefix_tree(h: int):
    """(nodes uint32 [n][8], tokens int32, upper uint32 [u][2], units uint32 [k][2]) of the handle's prefix tree."""
    sizes = np.zeros(4, dtype=np.int64)
    _check("domino_get_prefix_tree", lib().domino_get_prefix_tree(h, None, 0, None, 0, None, 0, None, 0, _ptr(sizes)))
    nodes = np.zeros((int(sizes[0]), 8), dtype=np.uint32)
    toks = np.zeros(int(sizes[1]), dtype=np.int32)
    upper = np.zeros((int(sizes[2]), 2), dtype=np.uint32)
    units = np.zeros((int(sizes[3]), 2), dtype=np.uint32)
    _check("domino_get_prefix_tree", lib().domino_get_prefix_tree(h, _ptr(nodes), nodes.shape[0], _ptr(toks),
                                                                   toks.shape[0], _ptr(upper), upper.shape[0],
                                                                   _ptr(units), units.shape[0], _ptr(sizes)))
    return nodes, toks, upper, units


def domino_precompute_table(h: int, next_dev, mask_dev, stream=None) -> None:
    _check("domino_precompute_table", lib().domino_precompute_table(h, _ptr(next_dev), _ptr(mask_dev),
                                                                     _stream(stream)))


def domino_step_mask(h: int, states_dev, stacks_dev, batch: int, mask_dev, next_dev=None, stream=None) -> None:
    _check("domino_step_mask", lib().domino_step_mask(h, _ptr(states_dev), _ptr(stacks_dev), int(batch),
                                                       _ptr(mask_dev), _ptr(next_dev), _stream(stream)))


def domino_mask_logits(h: int, logits_dev, dtype: int, batch: int, row_stride_elems: int, mask_dev, argmax_dev,
                       lse_dev=None, logprobs_dev=None, stream=None) -> None:
    _check("domino_mask_logits", lib().domino_mask_logits(
        h, _ptr(logits_dev), int(dtype), int(batch), int(row_stride_elems), _ptr(mask_dev), _ptr(argmax_dev),
        _ptr(lse_dev), _ptr(logprobs_dev), _stream(stream)))


def domino_advance(h: int, states_dev, stacks_dev, tokens_dev, batch: int, states_out, stacks_out=None,
                   stream=None) -> None:
    _check("domino_advance", lib().domino_advance(h, _ptr(states_dev), _ptr(stacks_dev), _ptr(tokens_dev),
                                                   int(batch), _ptr(states_out), _ptr(stacks_out), _stream(stream)))


def domino_step_decode(h: int, states_dev, stacks_dev, batch: int, logits_dev, dtype: int, row_stride_elems: int,
                       mask_dev, argmax_dev, lse_dev=None, logprobs_dev=None, states_out=None, stacks_out=None,
                       stream=None) -> None:
    _check("domino_step_decode", lib().domino_step_decode(
        h, _ptr(states_dev), _ptr(stacks_dev), int(batch), _ptr(logits_dev), int(dtype), int(row_stride_elems),
        _ptr(mask_dev), _ptr(argmax_dev), _ptr(lse_dev), _ptr(logprobs_dev), _ptr(states_out), _ptr(stacks_out),
        _stream(stream)))


def domino_mask_sample(h: int, logits_dev, dtype: int, batch: int, row_stride_elems: int, mask_dev,
                       temperature: float, seed: int, offset: int, tokens_dev, stream=None) -> None:
    _check("domino_mask_sample", lib().domino_mask_sample(
        h, _ptr(logits_dev), int(dtype), int(batch), int(row_stride_elems), _ptr(mask_dev), float(temperature),
        int(seed) & 0xFFFFFFFFFFFFFFFF, int(offset) & 0xFFFFFFFFFFFFFFFF, _ptr(tokens_dev), _stream(stream)))


def domino_opportunistic_step(h: int, logits_dev, dtype: int, batch: int, row_stride_elems: int, states_dev,
                              stacks_dev, mask_scratch_dev, tokens_dev, n_fallback_dev=None, stream=None) -> None:
    _check("domino_opportunistic_step", lib().domino_opportunistic_step(
        h, _ptr(logits_dev), int(dtype), int(batch), int(row_stride_elems), _ptr(states_dev), _ptr(stacks_dev),
        _ptr(mask_scratch_dev), _ptr(tokens_dev), _ptr(n_fallback_dev), _stream(stream)))


def domino_spec_update(h: int, counts_dev, best_dev, reached_dev, states_dev, stacks_dev, tokens_dev, batch: int,
                       stream=None) -> None:
    _check("domino_spec_update", lib().domino_spec_update(h, _ptr(counts_dev), _ptr(best_dev), _ptr(reached_dev),
                                                           _ptr(states_dev), _ptr(stacks_dev), _ptr(tokens_dev),
                                                           int(batch), _stream(stream)))


def domino_spec_propose(h: int, best_dev, reached_dev, states_dev, stacks_dev, batch: int, s: int, min_permille: int,
                        proposals_dev, n_prop_dev, chain_states_dev, chain_stacks_dev=None, stream=None) -> None:
    _check("domino_spec_propose", lib().domino_spec_propose(
        h, _ptr(best_dev), _ptr(reached_dev), _ptr(states_dev), _ptr(stacks_dev), int(batch), int(s),
        int(min_permille), _ptr(proposals_dev), _ptr(n_prop_dev), _ptr(chain_states_dev), _ptr(chain_stacks_dev),
        _stream(stream)))


def domino_spec_accept(h: int, proposals_dev, n_prop_dev, decoded_dev, chain_states_dev, chain_stacks_dev,
                       batch: int, s: int, n_accept_dev, tokens_out_dev=None, states_out_dev=None,
                       stacks_out_dev=None, stream=None) -> None:
    _check("domino_spec_accept", lib().domino_spec_accept(
        h, _ptr(proposals_dev), _ptr(n_prop_dev), _ptr(decoded_dev), _ptr(chain_states_dev), _ptr(chain_stacks_dev),
        int(batch), int(s), _ptr(n_accept_dev), _ptr(tokens_out_dev), _ptr(states_out_dev), _ptr(stacks_out_dev),
        _stream(stream)))


def domino_mask_logits_table(h: int, logits_dev, dtype: int, batch: int, row_stride_elems: int, table_mask_dev,
                             states_dev, argmax_dev, lse_dev=None, logprobs_dev=None, stream=None) -> None:
    _check("domino_mask_logits_table", lib().domino_mask_logits_table(
        h, _ptr(logits_dev), int(dtype), int(batch), int(row_stride_elems), _ptr(table_mask_dev), _ptr(states_dev),
        _ptr(argmax_dev), _ptr(lse_dev), _ptr(logprobs_dev), _stream(stream)))


def domino_advance_table(h: int, table_next_dev, states_dev, tokens_dev, batch: int, states_out, stream=None) -> None:
    _check("domino_advance_table", lib().domino_advance_table(h, _ptr(table_next_dev), _ptr(states_dev),
                                                               _ptr(tokens_dev), int(batch), _ptr(states_out),
                                                               _stream(stream)))


def domino_decode_step_host(h: int, logits_host, dtype: int, batch: int, states_host, stacks_host, tokens_host,
                            lse_host=None, stream=None) -> None:
    _check("domino_decode_step_host", lib().domino_decode_step_host(
        h, _ptr(logits_host), int(dtype), int(batch), _ptr(states_host), _ptr(stacks_host), _ptr(tokens_host),
        _ptr(lse_host), _stream(stream)))


def domino_mask_logits_noalloc(logits_dev, dtype: int, batch: int, n_tokens: int, row_stride_elems: int, mask_dev,
                               argmax_dev, lse_dev=None, logprobs_dev=None, stream=None) -> None:
    """domino_mask_logits for callers that cannot allocate: no handle, fixed scratch, batch <= 512."""
    _check("domino_mask_logits_noalloc", lib().domino_mask_logits_noalloc(
        _ptr(logits_dev), int(dtype), int(batch), int(n_tokens), int(row_stride_elems), _ptr(mask_dev),
        _ptr(argmax_dev), _ptr(lse_dev), _ptr(logprobs_dev), _stream(stream)))


def domino_get_device_error(h: int, stream=None) -> int:
    code = ctypes.c_int32(0)
    _check("domino_get_device_error", lib().domino_get_device_error(h, ctypes.byref(code), _stream(stream)))
    return code.value

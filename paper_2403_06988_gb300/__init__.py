"""DOMINO constrained decoding hot path on GB300 (sm_103a).

The compute lives in libdomino.so (C ABI in include/domino.h, kernels in
csrc/).  `_binding` exposes every entry point under its C name; `Domino`
below is a thin holder of one handle that allocates output tensors with torch
and forwards to those entry points.  There is no CPU fallback: without a
built libdomino.so the binding raises ImportError, and compute calls on a
handle created without a GPU raise DominoError(E_NO_DEVICE).
"""
from __future__ import annotations

from typing import Optional, Tuple

from . import _binding as B
from ._binding import DominoError, DTYPE_BF16, DTYPE_F32  # noqa: F401


class Domino:
    """One library handle: a vocabulary plus a scanner (+ bracket rules).

    fill_byte: None (default), or a byte value that every output buffer this
    holder allocates is filled with before the call that writes it.  A word a
    kernel leaves unwritten then keeps that pattern (0xAB bytes, say) instead
    of whatever the allocator handed back, so an exact comparison catches it.
    A debugging aid; it costs one fill per output.
    """

    fill_byte: Optional[int] = None

    def __init__(self, device: int = 0):
        self.device = device
        self.h = B.domino_create(device)

    def close(self):
        if self.h:
            B.domino_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- loads ---------------------------------------------------------------
    def load_vocab(self, vocab) -> None:
        B.domino_load_vocab(self.h, vocab.data, vocab.offsets, vocab.n_tokens, vocab.eos_id)

    def load_automaton(self, a) -> None:
        B.domino_load_automaton(self.h, a.delta, a.n_states, a.live, a.accepting, a.start, a.rules, None,
                                a.max_depth)

    @staticmethod
    def from_parts(automaton, vocab, device: int = 0) -> "Domino":
        d = Domino(device)
        d.load_vocab(vocab)
        d.load_automaton(automaton)
        return d

    def info(self) -> dict:
        return B.domino_get_info(self.h)

    def _empty(self, shape, dtype, device):
        import torch
        t = torch.empty(shape, dtype=dtype, device=device)
        if self.fill_byte is not None and t.numel():
            t.view(torch.uint8).fill_(self.fill_byte)
        return t

    # -- compute (torch tensors on this handle's device) -----------------------
    def step_mask(self, states, stacks=None, want_next: bool = False, out_mask=None, out_next=None,
                  stream=None):
        import torch
        info = self.info()
        b = states.shape[0]
        mask = out_mask if out_mask is not None else self._empty((b, info["n_words"]), torch.int32, states.device)
        nxt = out_next
        if want_next and nxt is None:
            nxt = self._empty((b, info["n_tokens"]), torch.int32, states.device)
        B.domino_step_mask(self.h, states, stacks, b, mask, nxt, stream)
        return mask, nxt

    def step_decode(self, states, stacks, logits, want_logprobs: bool = False, advance: bool = False, out_mask=None,
                    stream=None):
        """Mask step fused with the masked greedy decode: returns (mask, argmax, lse, logprobs or None).
        advance: states (and stacks) are then updated in place by the decoded tokens."""
        import torch
        b = states.shape[0]
        dtype = DTYPE_BF16 if logits.dtype == torch.bfloat16 else DTYPE_F32
        if dtype == DTYPE_F32 and logits.dtype != torch.float32:
            raise TypeError("logits must be float32 or bfloat16")
        if logits.stride(1) != 1:
            raise ValueError("logits rows must be contiguous")
        mask = out_mask if out_mask is not None else self._empty((b, self.info()["n_words"]), torch.int32,
                                                                 states.device)
        argmax = self._empty(b, torch.int32, states.device)
        lse = self._empty(b, torch.float32, states.device)
        lp = self._empty((b, self.info()["n_tokens"]), torch.float32, states.device) if want_logprobs else None
        B.domino_step_decode(self.h, states, stacks, b, logits.data_ptr(), dtype, logits.stride(0), mask, argmax, lse,
                             lp, states if advance else None, stacks if advance else None, stream)
        return mask, argmax, lse, lp

    def precompute_table(self, want_next: bool = True, want_mask: bool = True, stream=None):
        import torch
        info = self.info()
        dev = f"cuda:{self.device}"
        nxt = self._empty((info["n_states"], info["n_tokens"]), torch.int32, dev) if want_next else None
        mask = self._empty((info["n_states"], info["n_words"]), torch.int32, dev) if want_mask else None
        B.domino_precompute_table(self.h, nxt, mask, stream)
        return nxt, mask

    def mask_logits(self, logits, mask, want_lse: bool = True, want_logprobs: bool = False, n_tokens: Optional[int]
                    = None, out=None, stream=None) -> Tuple:
        import torch
        b = logits.shape[0]
        V = n_tokens if n_tokens is not None else self.info()["n_tokens"]
        dtype = DTYPE_BF16 if logits.dtype == torch.bfloat16 else DTYPE_F32
        if dtype == DTYPE_F32 and logits.dtype != torch.float32:
            raise TypeError("logits must be float32 or bfloat16")
        if logits.stride(1) != 1:
            raise ValueError("logits rows must be contiguous")
        argmax, lse, lp = out if out is not None else (None, None, None)
        if argmax is None:
            argmax = self._empty(b, torch.int32, logits.device)
        if want_lse and lse is None:
            lse = self._empty(b, torch.float32, logits.device)
        if want_logprobs and lp is None:
            lp = self._empty((b, V), torch.float32, logits.device)
        B.domino_mask_logits(self.h, logits.data_ptr(), dtype, b, logits.stride(0), mask, argmax,
                             lse if want_lse else None, lp if want_logprobs else None, stream)
        return argmax, (lse if want_lse else None), (lp if want_logprobs else None)

    def advance(self, states, stacks, tokens, states_out=None, stacks_out=None, stream=None):
        b = states.shape[0]
        so = states if states_out is None else states_out
        wo = stacks if stacks_out is None else stacks_out
        B.domino_advance(self.h, states, stacks, tokens, b, so, wo, stream)
        return so, wo

    def mask_sample(self, logits, mask, temperature: float, seed: int, offset: int, stream=None):
        """Gumbel-max draw per row from softmax(logits / T) over the allowed tokens (-1: none allowed)."""
        import torch
        b = logits.shape[0]
        dtype = DTYPE_BF16 if logits.dtype == torch.bfloat16 else DTYPE_F32
        if logits.stride(1) != 1:
            raise ValueError("logits rows must be contiguous")
        tokens = self._empty(b, torch.int32, logits.device)
        B.domino_mask_sample(self.h, logits, dtype, b, logits.stride(0), mask, temperature, seed, offset, tokens,
                             stream)
        return tokens

    def opportunistic_step(self, logits, states, stacks=None, stream=None):
        """Greedy tokens via opportunistic masking; returns (tokens, number of fallback rows as a tensor)."""
        import torch
        b = logits.shape[0]
        dtype = DTYPE_BF16 if logits.dtype == torch.bfloat16 else DTYPE_F32
        if logits.stride(1) != 1:
            raise ValueError("logits rows must be contiguous")
        W = self.info()["n_words"]
        scratch = self._empty((b, W), torch.int32, logits.device)
        tokens = self._empty(b, torch.int32, logits.device)
        n_fb = torch.zeros(1, dtype=torch.int32, device=logits.device)
        B.domino_opportunistic_step(self.h, logits, dtype, b, logits.stride(0), states, stacks, scratch, tokens, n_fb,
                                    stream)
        return tokens, n_fb

    def mask_logits_table(self, logits, table_mask, states, want_lse: bool = True, want_logprobs: bool = False,
                          stream=None) -> Tuple:
        """Table-driven mask + decode: row b's mask is table_mask[states[b]] (DFA only)."""
        import torch
        b = logits.shape[0]
        V = self.info()["n_tokens"]
        dtype = DTYPE_BF16 if logits.dtype == torch.bfloat16 else DTYPE_F32
        if logits.stride(1) != 1:
            raise ValueError("logits rows must be contiguous")
        argmax = self._empty(b, torch.int32, logits.device)
        lse = self._empty(b, torch.float32, logits.device) if want_lse else None
        lp = self._empty((b, V), torch.float32, logits.device) if want_logprobs else None
        B.domino_mask_logits_table(self.h, logits, dtype, b, logits.stride(0), table_mask, states, argmax, lse, lp,
                                   stream)
        return argmax, lse, lp

    def advance_table(self, table_next, states, tokens, states_out=None, stream=None):
        """Table-driven update: states_out[b] = table_next[states[b], tokens[b]] (DFA only)."""
        so = states if states_out is None else states_out
        B.domino_advance_table(self.h, table_next, states, tokens, states.shape[0], so, stream)
        return so

    def device_error(self, stream=None) -> int:
        return B.domino_get_device_error(self.h, stream)

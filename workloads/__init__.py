"""Seeded synthetic inputs for the beyond-mask joint attention.

This module is shared by the CPU oracle (tests) and the CUDA path (tests,
bench).  It holds only the workload shapes and the random-number recipe; it
contains none of the attention arithmetic.

Workload recipe (the paper's shapes, synthetic values):
  * one 1024x1024 image is 4096 latent tokens (Sec. 1); the live block is
    S = N_LT + N_X = 512 + 4096 = 4608 at 1024^2 (App. C, the one-reference
    example); a 512x512 image is 1024 tokens;
  * every reference image has the target's resolution (App. D, "Sampling":
    1024x1024 reference and output);
  * Q, K, V are bf16 with i.i.d. N(0, 1) elements, THD layout
    [tokens, heads, head_dim], requests packed back to back;
  * the prefill tensors hold each request's [ST; R] rows, the live tensors its
    [LT; X] rows (Sec. 3.3 order within each block).

Every tensor is drawn from torch's CPU Philox-free default generator
(mt19937-based ``torch.Generator``) seeded from (config seed, tensor name,
layer, step) through a fixed FNV-1a hash, so that both sides of a parity test
see the same bytes.
"""
from __future__ import annotations

import dataclasses
from typing import List, Sequence, Tuple

import torch


@dataclasses.dataclass(frozen=True)
class Request:
    """Segment lengths of one request: N_ST, N_LT, N_X, N_R (Sec. 3.1, 3.3)."""

    n_st: int
    n_lt: int
    n_x: int
    n_r: int

    @property
    def n_live(self) -> int:
        return self.n_lt + self.n_x

    @property
    def n_static(self) -> int:
        return self.n_st + self.n_r


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    num_heads: int
    head_dim: int
    requests: Tuple[Request, ...]
    seed: int

    @property
    def batch(self) -> int:
        return len(self.requests)

    def cu(self, lens: Sequence[int]) -> List[int]:
        out = [0]
        for n in lens:
            out.append(out[-1] + n)
        return out

    @property
    def cu_live(self) -> List[int]:
        return self.cu([r.n_live for r in self.requests])

    @property
    def cu_static(self) -> List[int]:
        return self.cu([r.n_static for r in self.requests])

    @property
    def n_anchor(self) -> List[int]:
        return [r.n_st for r in self.requests]

    @property
    def n_instr(self) -> List[int]:
        return [r.n_lt for r in self.requests]


def _w(name, h, d, reqs, seed):
    return Workload(name, h, d, tuple(Request(*r) for r in reqs), seed)


#: The five workloads: a tiny sanity case, a 512^2 edit with two references,
#: the 1024^2 five-reference headline shape, the 1024^2 reference sweep and a
#: ragged four-request serving batch.
TINY = _w("tiny_h4_d64", 4, 64, [(32, 64, 256, 256)], 0)
EDIT_512_2REF = _w("edit512_2ref", 24, 128, [(64, 256, 1024, 2 * 1024)], 1)
EDIT_1024_5REF = _w("edit1024_5ref", 24, 128, [(128, 512, 4096, 5 * 4096)], 2)
SWEEP_REFS = (1, 2, 5, 8, 10)
SWEEP_1024 = tuple(
    _w(f"edit1024_{k}ref", 24, 128, [(128, 512, 4096, k * 4096)], 2) for k in SWEEP_REFS
)
RAGGED_4REQ = _w(
    "ragged_4req",
    24,
    128,
    [
        (64, 256, 1024, 1 * 1024),
        (128, 512, 4096, 3 * 4096),
        (96, 384, 1024, 5 * 1024),
        (128, 512, 4096, 8 * 4096),
    ],
    3,
)

#: True classifier-free guidance (App. D, Sampling: gamma = 4 with a blank
#: negative prompt) runs a positive and a negative branch every step.  The
#: negative branch keeps the references and the target and has only the text
#: emptied (App. E): no live instruction tokens, and an anchor block of blank
#: text, so its reference cache differs from the positive branch's and is a
#: request of its own.  Both branches run as two requests of one ragged batch,
#: one launch per call.
CFG_1024_5REF = _w("cfg_edit1024_5ref", 24, 128, [(128, 512, 4096, 5 * 4096), (128, 0, 4096, 5 * 4096)], 4)
CFG_SMALL = _w("cfg_small", 4, 128, [(32, 64, 512, 1024), (32, 0, 512, 1024)], 5)

ALL = {w.name: w for w in (TINY, EDIT_512_2REF, EDIT_1024_5REF, RAGGED_4REQ, CFG_1024_5REF, CFG_SMALL) + SWEEP_1024}


def _fnv1a(text: str) -> int:
    h = 0xCBF29CE484222325
    for b in text.encode():
        h ^= b
        h = (h * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h & 0x7FFFFFFFFFFFFFFF


def tensor_seed(seed: int, name: str, layer: int = 0, step: int = 0) -> int:
    return _fnv1a(f"{seed}/{name}/{layer}/{step}")


def randn_bf16(shape, seed: int, name: str, layer: int = 0, step: int = 0) -> torch.Tensor:
    """bf16 N(0,1) tensor on the CPU (fp32 draw rounded to nearest-even bf16)."""
    g = torch.Generator(device="cpu")
    g.manual_seed(tensor_seed(seed, name, layer, step))
    return torch.randn(*shape, generator=g, dtype=torch.float32).to(torch.bfloat16)


def static_qkv(w: Workload, layer: int = 0):
    """[ST; R] rows of every request, THD bf16: q, k, v."""
    n = w.cu_static[-1]
    shape = (n, w.num_heads, w.head_dim)
    return tuple(randn_bf16(shape, w.seed, f"static_{t}", layer) for t in "qkv")


def live_qkv(w: Workload, layer: int = 0, step: int = 0):
    """[LT; X] rows of every request for one denoising step, THD bf16."""
    n = w.cu_live[-1]
    shape = (n, w.num_heads, w.head_dim)
    return tuple(randn_bf16(shape, w.seed, f"live_{t}", layer, step) for t in "qkv")


def bf16_bits(t: torch.Tensor):
    """Raw bf16 bit patterns of a CPU tensor as a numpy uint16 array."""
    return t.contiguous().view(torch.int16).numpy().view("uint16")


def random_requests(rng, batch: int, max_len: int = 200, allow_empty: bool = True):
    """Ragged small requests for parity sweeps (lengths include 0, 1 and odd)."""
    lo = 0 if allow_empty else 1
    reqs = []
    for _ in range(batch):
        n_st = int(rng.integers(lo, 40))
        n_lt = int(rng.integers(lo, 60))
        n_x = int(rng.integers(1, max_len))
        n_r = int(rng.integers(1, max_len))
        reqs.append(Request(n_st, n_lt, n_x, n_r))
    return tuple(reqs)

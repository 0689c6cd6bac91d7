"""Layered dependency graph of App. A (test infrastructure only).

A layer-shared block mask M over a block set V; ``attends(q, k)`` says that
block q attends to block k (the paper writes M[k, q] = 1 for the same
relation, App. A Eq. blockrec).  Unrolling across depth gives nodes (b, l) for l = 0..L,
residual edges (b, l-1) -> (b, l) and attention edges (k, l-1) -> (q, l)
whenever q attends k.

  StructCacheable(R)    <=>  (X, 0) reaches no (R, l), l = 1..L  (Eq. def-cache)
  LiveTextReachable(R)  <=>  (LT, l) reaches (R, m) for some 1 <= l < m <= L
                                                        (Eq. def-instr)
Theorem 1: with L >= 2, a layer-shared mask on {LT, X, R} and LT attending X,
no mask satisfies both.
"""
from __future__ import annotations

import itertools
from typing import Callable, Dict, Iterable, Set, Tuple

Node = Tuple[str, int]


def reachable_from(blocks: Iterable[str], attends: Callable[[str, str], bool], src: Node,
                   depth: int) -> Set[Node]:
    blocks = tuple(blocks)
    seen = {src}
    frontier = [src]
    while frontier:
        b, l = frontier.pop()
        if l >= depth:
            continue
        succ = [(b, l + 1)] + [(q, l + 1) for q in blocks if attends(q, b)]
        for n in succ:
            if n not in seen:
                seen.add(n)
                frontier.append(n)
    return seen


def struct_cacheable(blocks, attends, depth: int) -> bool:
    r = reachable_from(blocks, attends, ("X", 0), depth)
    return not any(("R", l) in r for l in range(1, depth + 1))


def live_text_reachable(blocks, attends, depth: int) -> bool:
    for l in range(1, depth + 1):
        r = reachable_from(blocks, attends, ("LT", l), depth)
        if any(("R", m) in r for m in range(l + 1, depth + 1)):
            return True
    return False


def instruction_reaches_reference(blocks, attends, depth: int) -> bool:
    """The static instruction carrier reaches R (the path Sec. 3.3 adds)."""
    r = reachable_from(blocks, attends, ("ST", 0), depth)
    return any(("R", l) in r for l in range(1, depth + 1))


def all_masks(blocks) -> Iterable[Dict[Tuple[str, str], bool]]:
    pairs = [(q, k) for q in blocks for k in blocks]
    for bits in itertools.product((False, True), repeat=len(pairs)):
        yield dict(zip(pairs, bits))

"""Work accounting for the hot path: unmasked attention units and FLOPs.

One unit is one (query row, key) interaction of one head; its algorithmic cost
is 4 * head_dim FLOPs (2d for the score, 2d for the P.V product).  Per
request, with S = N_LT + N_X (App. C, "Derivation"):
  prefill units  (N_ST + N_R)^2                (Eq. cost-pre; the alternative
                 anchor reading: N_ST^2 + N_R (N_ST + N_R))
  step units     S (S + N_R)                   (Eq. cost-step; + S N_ST in the
                 alternative reading, whose live rows also see the anchors)
  full units     (S + N_R)^2                   (C_full / T)
and the modelled T-step ratio is T C_full-step / (C_pre + T C_step) (Eq. speedup).
"""
from __future__ import annotations


def _lens(req):
    return req.n_st, req.n_lt, req.n_x, req.n_r


def prefill_units(requests, mode="beyond"):
    u = 0
    for r in requests:
        n_st, _, _, n_r = _lens(r)
        if mode == "beyond_alt":
            u += n_st * n_st + n_r * (n_st + n_r)
        else:
            u += (n_st + n_r) ** 2
    return u


def step_units(requests, mode="beyond"):
    u = 0
    for r in requests:
        n_st, n_lt, n_x, n_r = _lens(r)
        s = n_lt + n_x
        u += s * (s + n_r + (n_st if mode == "beyond_alt" else 0))
    return u


def full_units(requests):
    return sum((r.n_lt + r.n_x + r.n_r) ** 2 for r in requests)


def flops(units, num_heads, head_dim):
    return 4 * head_dim * num_heads * units


def modelled_ratio(requests, T=40, mode="beyond"):
    """Interaction-count speedup of the cache over full attention over T steps."""
    return T * full_units(requests) / (prefill_units(requests, mode) + T * step_units(requests, mode))


def measured_ratio(t_full_step, t_prefill, t_step, T=40):
    """The same ratio from measured per-call times: T t_full / (t_prefill + T t_step)."""
    return T * t_full_step / (t_prefill + T * t_step)


def cache_bytes(requests, num_heads, head_dim, mode="beyond"):
    """Bytes of one layer's cached K and V (bf16)."""
    rows = sum(r.n_r + (r.n_st if mode == "beyond_alt" else 0) for r in requests)
    return 2 * rows * num_heads * head_dim * 2

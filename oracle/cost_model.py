"""Attention-interaction cost model of App. C (test infrastructure only).

One unit is one query-key interaction.  With S = N_X + N_LT:
  C_pre  = (N_R + N_ST)^2                         (Eq. cost-pre)
  C_step = S (N_R + S)                            (Eq. cost-step)
  C_ours = C_pre + T C_step                       (Eq. cost-ours)
  C_full = T (N_R + S)^2
  R      = C_full / C_ours                        (Eq. speedup)
  R'(u)  = T u [2 a (u + a) + T S u] / D(u)^2,  u = N_R + S, a = N_ST - S,
           D(u) = (u + a)^2 + T S u               (Eqs. speedup-u, speedup-deriv)
  R_asym ~ T N_R / (N_R + T S)                    (Eq. speedup-asymptotic)
  Delta_A_ST = 2 N_R N_ST + N_ST^2                (Eq. anchor-overhead, Sec. 3.3)
"""
from __future__ import annotations


def c_pre(n_r, n_st):
    return (n_r + n_st) ** 2


def c_step(n_r, s):
    return s * (n_r + s)


def c_ours(n_r, n_st, s, T):
    return c_pre(n_r, n_st) + T * c_step(n_r, s)


def c_full(n_r, s, T):
    return T * (n_r + s) ** 2


def speedup(n_r, n_st, s, T):
    return c_full(n_r, s, T) / c_ours(n_r, n_st, s, T)


def speedup_of_u(u, n_st, s, T):
    a = n_st - s
    return T * u * u / ((u + a) ** 2 + T * s * u)


def speedup_derivative_u(u, n_st, s, T):
    a = n_st - s
    D = (u + a) ** 2 + T * s * u
    return T * u * (2 * a * (u + a) + T * s * u) / D ** 2


def speedup_asymptotic(n_r, s, T):
    return T * n_r / (n_r + T * s)


def anchor_overhead(n_r, n_st):
    return 2 * n_r * n_st + n_st ** 2


def flops_per_unit(head_dim):
    """Unmasked FLOPs of one (query, key) interaction for one head: 2d (QK^T) + 2d (PV)."""
    return 4 * head_dim

"""A rigorous bound on how far the head step computed with bf16 layer inputs
and fp32 accumulation (the library's dataflow, and the oracle's
clover_head_step reading of it) can fall from the same step in exact
arithmetic (oracle.clover_head_step_exact).

Errors are carried as 2-norms of each row's error vector, layer by layer
(u = 2^-8, the unit roundoff of bf16 with round to nearest even; u32 = 2^-24,
that of fp32):
  - the embedding is an fp32 normalisation (relative error at most
    (H + 8) u32 per element: a sum of H squares, a square root, a reciprocal
    and a product) rounded once to bf16: E_e = (u + (H + 8) u32 (1 + u)) |e|;
  - a layer y = W x with an input error of norm E_x moves y by at most
    ||W||_2 E_x (the spectral norm);
  - it multiplies bf16 values exactly and sums K products in fp32: element i
    within gamma_K (|W| |x|)_i, gamma_K = 2 K u32 (twice the classical
    (K-1) u32, for any summation order and a split of K), so in norm within
    gamma_K || |W| ||_2 (||x|| + E_x);
  - a residual is added in fp32 (u32 relative) and a bf16 output is rounded
    once (u relative), each adding at most that fraction of the output's norm;
  - silu(v) = v / (1 + 2^(-v log2 e)) is 1.1-Lipschitz (its derivative lies
    in [-0.1, 1.1]) and is evaluated in fp32 with an approximate exponent,
    relative error at most 2^-22 + (1.5 |v| + 4) u32.
A logit is one row of the LM head against z, so by Cauchy-Schwarz its error
is at most ||w_lm[v]||_2 E_z plus its own fp32 summation.  Every step is an
upper bound, so both the library and the bf16-reading oracle must meet E; a
dropped term, a wrong sign or a transposed weight moves logits by amounts of
the order of the logits themselves and breaks it.
"""

from __future__ import annotations

import torch

U = 2.0 ** -8
U32 = 2.0 ** -24


def _spec(W: torch.Tensor) -> float:
    return float(torch.linalg.matrix_norm(W, ord=2))


def head_step_bound(h, w_lm, w_v, w_o, w_1, ex) -> torch.Tensor:
    """E [R, V]: the bound on |logit - exact logit|, from the exact step's
    intermediates ``ex`` (oracle.clover_head_step_exact)."""
    H = h.shape[1]
    g = 2.0 * H * U32                                  # every layer here sums H products
    nrm = lambda t: t.double().norm(dim=-1)            # per-row 2-norm [R]
    Wv, Wo, W1, Wlm = (w.double() for w in (w_v, w_o, w_1, w_lm))

    def layer(E_x, x, W, y):
        """Error norm of y = W x_k before its output rounding."""
        return _spec(W) * E_x + g * _spec(W.abs()) * (nrm(x) + E_x)

    E_e = (U + (H + 8) * U32 * (1 + U)) * nrm(ex["e"])

    E_a = layer(E_e, ex["e"], Wv, ex["v"])
    E_a = E_a + U * (nrm(ex["v"]) + E_a)                # bf16 output

    E_h = layer(E_a, ex["v"], Wo, ex["attn"])
    E_h = E_h + U32 * (nrm(ex["h"]) + E_h)              # residual add
    E_h = E_h + U * (nrm(ex["h"]) + E_h)                # bf16 output

    u = ex["h"] @ W1.T
    E_u = layer(E_h, ex["h"], W1, u)
    silu = u / (1.0 + torch.exp(-u))
    rel = 2.0 ** -22 + (1.5 * (u.abs().amax(dim=-1) + E_u) + 4) * U32
    E_s = 1.1 * E_u + rel * (nrm(silu) + 1.1 * E_u)
    E_z = E_h + E_s
    E_z = E_z + U32 * (nrm(ex["z"]) + E_z)              # residual add
    E_z = E_z + U * (nrm(ex["z"]) + E_z)                # bf16 output

    # logit (r, v) = w_lm[v] . z_k[r]: its error and its fp32 sum
    row = Wlm.norm(dim=-1)                             # [V]
    E_l = E_z[:, None] * row[None, :]
    E_l = E_l + g * (ex["z"].abs() @ Wlm.abs().T + E_z[:, None] * row[None, :])
    return E_l + U32 * (ex["logits"].abs() + E_l)

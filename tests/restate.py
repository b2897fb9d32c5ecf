"""Independent fp64 restatement of the encoder with ``torch.nn.functional`` (CPU).

Used only to pin the oracle: it shares no code with ``oracle/`` and states each step
with library routines (reshape/permute patchify, ``F.linear``, ``F.layer_norm``,
``F.scaled_dot_product_attention``, ``F.gelu``) instead of loops.  Incremental steps
are stated with masks: the full K/V of a layer is ``where(updated, new, cached)``
(Eq. 5) and only updated rows run the block (Sec. III-B).
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F

from paper_2607_12287_gb300 import synth


def weights64(shape, w_u16) -> dict:
    parts = synth.split_weights(shape, np.asarray(w_u16, np.uint16))
    return {k: torch.from_numpy(synth.bf16_bits_to_f32(v).astype(np.float64)).reshape(v.shape)
            for k, v in parts.items()}


def embed(shape, W, frame) -> torch.Tensor:
    """frame uint8 [H, W, 3] -> patch embeddings [N, D] (before position embedding)."""
    P, gh, gw = shape.patch, shape.grid_h, shape.grid_w
    x = torch.from_numpy(np.asarray(frame).astype(np.float64)) - 128.0
    patches = x.reshape(gh, P, gw, P, 3).permute(0, 2, 1, 3, 4).reshape(gh * gw, P * P * 3)
    return F.linear(patches, W["W_pe"], W["b_pe"])


def _gelu(x, shape):
    return F.gelu(x, approximate="tanh" if shape.gelu == synth.GELU_TANH else "none")


def _attend(q, K, V, H):
    m, D = q.shape
    n = K.shape[0]
    dh = D // H
    qh = q.reshape(m, H, dh).transpose(0, 1)
    kh = K.reshape(n, H, dh).transpose(0, 1)
    vh = V.reshape(n, H, dh).transpose(0, 1)
    o = F.scaled_dot_product_attention(qh[None], kh[None], vh[None])[0]
    return o.transpose(0, 1).reshape(m, D)


def run_rows(shape, W, e, mask, K, V, tokens):
    """Runs the blocks for the tokens where ``mask`` is true; K, V [L, N, D] and tokens
    [N, D] are the cached state, updated in place copies that are returned."""
    D, H, eps = shape.dim, shape.heads, shape.ln_eps
    K, V, tokens = K.clone(), V.clone(), tokens.clone()
    sel = torch.nonzero(torch.as_tensor(mask)).flatten()
    x = (e + W["pos"])[sel]
    for l in range(shape.depth):
        p = lambda n: W[f"l{l}.{n}"]
        xn = F.layer_norm(x, (D,), p("ln1_g"), p("ln1_b"), eps)
        q, k, v = F.linear(xn, p("W_qkv"), p("b_qkv")).split(D, dim=1)
        K[l] = K[l].index_put((sel,), k)
        V[l] = V[l].index_put((sel,), v)
        x = x + F.linear(_attend(q, K[l], V[l], H), p("W_o"), p("b_o"))
        hdn = _gelu(F.linear(F.layer_norm(x, (D,), p("ln2_g"), p("ln2_b"), eps),
                             p("W_1"), p("b_1")), shape)
        x = x + F.linear(hdn, p("W_2"), p("b_2"))
    tokens[sel] = F.layer_norm(x, (D,), W["lnf_g"], W["lnf_b"], eps)
    return K, V, tokens


def full(shape, W, frame):
    """Full encode of one view: (tokens [N, D], K [L, N, D], V [L, N, D], e [N, D])."""
    N, D, L = shape.n_tokens, shape.dim, shape.depth
    e = embed(shape, W, frame)
    K = torch.zeros(L, N, D, dtype=torch.float64)
    V = torch.zeros_like(K)
    tok = torch.zeros(N, D, dtype=torch.float64)
    K, V, tok = run_rows(shape, W, e, torch.ones(N, dtype=torch.bool), K, V, tok)
    return tok, K, V, e


def layer0_keys(shape, W, e):
    """Eq. 3 key vectors of every token in fp64: W_K LN1(e + pos) + b_K."""
    D = shape.dim
    xn = F.layer_norm(e + W["pos"], (D,), W["l0.ln1_g"], W["l0.ln1_b"], shape.ln_eps)
    return F.linear(xn, W["l0.W_qkv"][D:2 * D], W["l0.b_qkv"][D:2 * D])


def run_rows_mlp_all(shape, W, e, mask, K, V, A):
    """The MLP-on-all-tokens reading (Sec. III-B, after Eq. 5): attention for the tokens
    where ``mask`` is true only (their K/V and attention-block outputs replace the cached
    ones in K, V, A [L, N, D]); every token then takes the residual addition with its
    attention-block output (cached for reused tokens), LN2 + MLP, and the final LN.
    Returns (K, V, A, tokens [N, D]) as new tensors."""
    D, H, eps = shape.dim, shape.heads, shape.ln_eps
    K, V, A = K.clone(), V.clone(), A.clone()
    sel = torch.nonzero(torch.as_tensor(mask)).flatten()
    x = e + W["pos"]
    for l in range(shape.depth):
        p = lambda n: W[f"l{l}.{n}"]
        xn = F.layer_norm(x[sel], (D,), p("ln1_g"), p("ln1_b"), eps)
        q, k, v = F.linear(xn, p("W_qkv"), p("b_qkv")).split(D, dim=1)
        K[l] = K[l].index_put((sel,), k)
        V[l] = V[l].index_put((sel,), v)
        A[l] = A[l].index_put((sel,), F.linear(_attend(q, K[l], V[l], H), p("W_o"), p("b_o")))
        x = x + A[l]
        x = x + F.linear(_gelu(F.linear(F.layer_norm(x, (D,), p("ln2_g"), p("ln2_b"), eps),
                                        p("W_1"), p("b_1")), shape), p("W_2"), p("b_2"))
    return K, V, A, F.layer_norm(x, (D,), W["lnf_g"], W["lnf_b"], eps)


def full_mlp_all(shape, W, frame):
    """Full encode under the MLP-on-all-tokens reading: (tokens, K, V, A, e)."""
    N, D, L = shape.n_tokens, shape.dim, shape.depth
    e = embed(shape, W, frame)
    Z = torch.zeros(L, N, D, dtype=torch.float64)
    K, V, A, tok = run_rows_mlp_all(shape, W, e, torch.ones(N, dtype=torch.bool), Z, Z, Z)
    return tok, K, V, A, e

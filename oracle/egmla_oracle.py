"""Plain fp64 CPU oracle for EG-MLA decode (test infrastructure only).

This module is the parity reference for the CUDA path.  Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
it; the library itself never does.  It shares no code with the CUDA path: the
only common module is the seeded input generator, which holds none of the
method's arithmetic.

Everything is computed in float64 from the stored input bits (bf16 widened
exactly), with no blocking, splitting, fusion or absorption beyond what each
function's docstring states.  Citations are to the EG-MLA paper (arXiv
2509.16686): section 3 ("Embedding Gated MLA", Eqs. 1-5), Appendix C (full
formulas, Eqs. 1-14), Appendix E (the PyTorch listing), Table 5 and the Appendix
F cache table.

Reading of the gate placement (the paper is not self-consistent, see the
repository design notes): the hot path gates the compressed latent,
``c~ = LN_{d_c}(c (*) g)``, with ``g = G[id]`` the precomputed gate row of the
inference variant EG-MLA-A (Section 5.2).  The paper-literal form that gates the
up-projected keys/values (Eq. 5 applied after Eq. 2, as in the listing) is kept
as ``decode_r0`` for documentation.

Parity status: every function here is pinned by the tests in
``tests/test_oracle_pins.py`` (library routines, closed forms, invariants, the
paper's printed cache sizes).  The attention-layer step (``layer_step``,
``layer_decode``) is pinned by decoding a sequence one token at a time against
one causal forward pass over the whole sequence written from the listing, and
its RoPE, RMSNorm and bf16 storage against the corresponding torch routines.
``prefill`` (every position of a prompt at once) is pinned row by row against
``decode_unabsorbed`` on the cache holding the prompt up to that row, against
torch's causal scaled_dot_product_attention where the projections are
identities, by a one-token closed form, the causal running mean at q = 0, and
causality and prompt-independence invariants.  ``decode_r0`` (the paper
prints no numeric example of it) is pinned against a PyTorch re-expression of the paper's listing, a single-token
closed form, invariance under permuting cached positions, and its reduction to
the latent-gated form when the joint up-projection is the identity.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Iterable, Optional

import numpy as np


# --------------------------------------------------------------------------
# storage
# --------------------------------------------------------------------------
def widen(x: np.ndarray, dtype: str) -> np.ndarray:
    """Stored values -> float64.  bf16 arrives as uint16 bit patterns."""
    if dtype == "bf16":
        b = np.ascontiguousarray(x, dtype=np.uint16)
        return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return np.asarray(x, dtype=np.float64)


def softmax_scale(d) -> float:
    """Attention scale 1/sqrt(d_h + d_h^R) (Appendix C Eq. 13; the listing's SDPA
    default over q of width d_nope + d_rope), unless the dims fix another one."""
    if d.softmax_scale > 0:
        return float(d.softmax_scale)
    return 1.0 / math.sqrt(d.d_nope + d.d_rope)


# --------------------------------------------------------------------------
# paged latent cache (Table 5: the cache holds d_c + d_h^R values per token)
# --------------------------------------------------------------------------
def paged_position(block_table: np.ndarray, b: int, j: int, page_size: int):
    """Logical position j of sequence b -> (physical page, slot in page)."""
    return int(block_table[b, j // page_size]), j % page_size


def gather_sequence(pool: np.ndarray, block_table: np.ndarray, b: int, length: int,
                    page_size: int) -> np.ndarray:
    """Rows 0..length-1 of sequence b, read through the block table one by one."""
    rows = []
    for j in range(length):
        page, slot = paged_position(block_table, b, j, page_size)
        rows.append(pool[page, slot])
    if not rows:
        return pool[:0, 0]
    return np.stack(rows, axis=0)


def append_latent(c_pool, kr_pool, id_pool, c_new, kr_new, ids_new, block_table, positions,
                  page_size: int):
    """Host scatter of each sequence's new token into its cache slot (Appendix C Eq. 1
    and Eq. 10 produce c^KV and the rotated k^R; those two, plus the token id, are
    what the cache keeps).  Returns new arrays; inputs are not modified.
    A negative position means "nothing to append" for that sequence."""
    c_pool, kr_pool = c_pool.copy(), kr_pool.copy()
    id_pool = None if id_pool is None else id_pool.copy()
    for b in range(positions.shape[0]):
        pos = int(positions[b])
        if pos < 0:
            continue
        page, slot = paged_position(block_table, b, pos, page_size)
        c_pool[page, slot] = c_new[b]
        kr_pool[page, slot] = kr_new[b]
        if id_pool is not None and ids_new is not None:
            id_pool[page, slot] = ids_new[b]
    return c_pool, kr_pool, id_pool


# --------------------------------------------------------------------------
# gate (Section 3 Eqs. 3-5; inference variant EG-MLA-A in Section 5.2)
# --------------------------------------------------------------------------
def gate_table_from_embedding(emb: np.ndarray, w_ue: np.ndarray) -> np.ndarray:
    """G[i] = W^UE Emb(i) for every vocabulary entry (Eqs. 3-4), precomputed once
    as EG-MLA-A does at model-load time.  emb [V, d_e], w_ue [d_gate, d_e]."""
    return np.asarray(emb, np.float64) @ np.asarray(w_ue, np.float64).T


def layer_norm(x: np.ndarray, gamma: np.ndarray, beta: np.ndarray, eps: float) -> np.ndarray:
    """LN over the last axis with biased variance and affine gamma/beta (the listing's
    nn.LayerNorm with its default eps=1e-5)."""
    mean = x.mean(axis=-1, keepdims=True)
    var = ((x - mean) ** 2).mean(axis=-1, keepdims=True)
    return (x - mean) / np.sqrt(var + eps) * gamma + beta


def gated_latent(c: np.ndarray, g: np.ndarray, gamma, beta, eps: float) -> np.ndarray:
    """Eq. 5 in latent space: c~ = LN(c (*) g); the Hadamard product comes first."""
    return layer_norm(c * g, gamma, beta, eps)


def gated_latent_no_norm(c: np.ndarray, g: np.ndarray) -> np.ndarray:
    """Section 4.4 ablation "remove LayerNorm" (Table 'Ablation on Embedding
    Gating'): Eq. 5 without its LayerNorm, c~ = c (*) g."""
    return c * g


def gated_latent_added(c: np.ndarray, g: np.ndarray, gamma, beta, eps: float) -> np.ndarray:
    """Section 4.4 ablation "replace (*) with addition": c~ = LN(c + g)."""
    return layer_norm(c + g, gamma, beta, eps)


def gate_latents(c: np.ndarray, g: np.ndarray, gamma, beta, eps: float, op: str) -> np.ndarray:
    """The gated latent of gate operation `op`: "mul_ln" (the method, Eq. 5),
    "mul" or "add_ln" (the two ablations of Section 4.4)."""
    if op == "mul_ln":
        return gated_latent(c, g, gamma, beta, eps)
    if op == "mul":
        return gated_latent_no_norm(c, g)
    if op == "add_ln":
        return gated_latent_added(c, g, gamma, beta, eps)
    raise ValueError(f"unknown gate operation {op!r}")


# --------------------------------------------------------------------------
# attention for one decode query (Appendix C Eqs. 11-13)
# --------------------------------------------------------------------------
def softmax(s: np.ndarray) -> np.ndarray:
    """Max-subtracted softmax over the last axis.  An empty axis gives an empty result."""
    if s.shape[-1] == 0:
        return s.copy()
    m = s.max(axis=-1, keepdims=True)
    e = np.exp(s - m)
    return e / e.sum(axis=-1, keepdims=True)


def _sequence_latents(case, b: int, gate: bool):
    """(c~ [L, d_c], k^R [L, d_r]) of sequence b after the new token is appended."""
    d = case.dims
    L = int(case.seq_lens[b])
    c_pool, kr_pool, id_pool = appended_pools(case)
    c = widen(gather_sequence(c_pool, case.block_table, b, L, d.page_size), d.dtype)
    kr = widen(gather_sequence(kr_pool, case.block_table, b, L, d.page_size), d.dtype)
    if gate:
        ids = gather_sequence(id_pool, case.block_table, b, L, d.page_size).astype(np.int64)
        g = widen(case.gate_table, d.dtype)[ids] if L > 0 else np.zeros((0, d.d_c))
        c_t = gate_latents(c, g, np.asarray(case.ln_gamma, np.float64), np.asarray(case.ln_beta, np.float64),
                           d.ln_eps, getattr(d, "gate_op", "mul_ln"))
    else:
        c_t = c
    return c_t, kr


def appended_pools(case):
    """The cache after this step's append (computed once per case and kept on it)."""
    got = getattr(case, "_oracle_appended", None)
    if got is None:
        d = case.dims
        got = append_latent(case.c_pool, case.kr_pool, case.id_pool, case.c_new, case.kr_new,
                            case.ids_new, case.block_table, case.positions(), d.page_size)
        case._oracle_appended = got
    return got


def head_probs_unabsorbed(case, b: int, h: int, gate: Optional[bool] = None):
    """Softmax weights p_j of head h of sequence b over its L_b cached positions.

    Keys are k_j = [W_UK,h c~_j ; k^R_j] (Eqs. 6 and 12, the RoPE key shared by all
    heads and not gated), the query is q = [q^C ; q^R] (Eq. 11) and the scale is
    1/sqrt(d_h + d_h^R) (Eq. 13)."""
    d = case.dims
    gate = d.gate if gate is None else gate
    c_t, kr = _sequence_latents(case, b, gate)
    qv = widen(case.q[b, h], d.dtype)
    w_uk = widen(case.w_uk[h], d.dtype)               # [d_n, d_c]
    k_c = c_t @ w_uk.T                                 # [L, d_n]   (Eq. 2 + split, Eq. 6)
    k = np.concatenate([k_c, kr], axis=1)              # [L, d_n + d_r] (Eq. 12)
    s = (k @ qv) * softmax_scale(d)                           # (Eq. 13)
    return softmax(s), c_t


def decode_unabsorbed(case, batches: Optional[Iterable[int]] = None,
                      heads: Optional[Iterable[int]] = None, gate: Optional[bool] = None) -> np.ndarray:
    """u_{t,i} = sum_j softmax_j(q_i . k_{j,i} / sqrt(d_h + d_h^R)) v_{j,i}   (Eq. 13)

    with v_{j,i} = W_UV,i c~_j (Eq. 2 + split, Eq. 6): naive per-head MLA that
    up-projects every cached latent.  Returns [B, H, d_v] float64 (rows of
    unselected batches/heads are NaN).  A sequence of length 0 gives zeros."""
    d = case.dims
    gate = d.gate if gate is None else gate
    B, H = case.batch, d.num_heads
    out = np.full((B, H, d.d_v), np.nan)
    bs = range(B) if batches is None else list(batches)
    hs = range(H) if heads is None else list(heads)
    for b in bs:
        L = int(case.seq_lens[b])
        if L == 0:
            out[b, list(hs)] = 0.0
            continue
        c_t, kr = _sequence_latents(case, b, gate)
        for h in hs:
            qv = widen(case.q[b, h], d.dtype)
            w_uk = widen(case.w_uk[h], d.dtype)
            w_uv = widen(case.w_uv[h], d.dtype)
            k = np.concatenate([c_t @ w_uk.T, kr], axis=1)
            v = c_t @ w_uv.T                             # [L, d_v]
            p = softmax((k @ qv) * softmax_scale(d))
            out[b, h] = p @ v
    return out


def decode_absorbed(case, batches=None, heads=None, gate: Optional[bool] = None) -> np.ndarray:
    """The same output computed in weight-absorbed form: q^ = W_UK,h^T q^C scores the
    shared latent directly (q.(W c~) = (W^T q).c~), the latent-space output
    o = sum_j p_j c~_j is formed first and W_UV,h is applied once at the end."""
    d = case.dims
    gate = d.gate if gate is None else gate
    B, H = case.batch, d.num_heads
    out = np.full((B, H, d.d_v), np.nan)
    bs = range(B) if batches is None else list(batches)
    hs = range(H) if heads is None else list(heads)
    for b in bs:
        L = int(case.seq_lens[b])
        if L == 0:
            out[b, list(hs)] = 0.0
            continue
        c_t, kr = _sequence_latents(case, b, gate)
        for h in hs:
            qv = widen(case.q[b, h], d.dtype)
            q_nope, q_rope = qv[:d.d_nope], qv[d.d_nope:]
            q_hat = widen(case.w_uk[h], d.dtype).T @ q_nope          # [d_c]
            s = (c_t @ q_hat + kr @ q_rope) * softmax_scale(d)
            o_lat = softmax(s) @ c_t                                 # [d_c]
            out[b, h] = widen(case.w_uv[h], d.dtype) @ o_lat
    return out


def decode_r0(case, w_ukv_full: Optional[np.ndarray] = None, gate_r0: Optional[np.ndarray] = None,
              ln_gamma_r0=None, ln_beta_r0=None, batches=None) -> np.ndarray:
    """Paper-literal gating (Eq. 5 after Eq. 2, as the Appendix E listing does):
    kv~ = LN_{H(d_n+d_v)}((W^UKV c) (*) g) over all heads at once, split per head
    into k^C, v^C (Eq. 6), then Eqs. 11-13.  ``gate_r0`` [V, H(d_n+d_v)] is the
    precomputed gate in that space and must be given.  W^UKV defaults to stacking
    W_UK,h and W_UV,h per head (keys, then values, head by head, the row order
    of the joint up-projection in Appendix E).
    Returns [B, H, d_v]."""
    d = case.dims
    B, H, dn, dv = case.batch, d.num_heads, d.d_nope, d.d_v
    if w_ukv_full is None:
        w_ukv_full = np.concatenate([widen(case.w_uk, d.dtype), widen(case.w_uv, d.dtype)], axis=1)
        w_ukv_full = w_ukv_full.reshape(H * (dn + dv), d.d_c)
    width = H * (dn + dv)
    gamma = np.ones(width) if ln_gamma_r0 is None else np.asarray(ln_gamma_r0, np.float64)
    beta = np.zeros(width) if ln_beta_r0 is None else np.asarray(ln_beta_r0, np.float64)
    out = np.full((B, H, dv), np.nan)
    bs = range(B) if batches is None else list(batches)
    for b in bs:
        L = int(case.seq_lens[b])
        if L == 0:
            out[b] = 0.0
            continue
        c_raw, kr = _sequence_latents(case, b, gate=False)
        ids = gather_sequence(appended_pools(case)[2], case.block_table, b, L, d.page_size)
        kv = c_raw @ w_ukv_full.T                                   # [L, H(dn+dv)]  Eq. 2
        kv = layer_norm(kv * np.asarray(gate_r0, np.float64)[ids], gamma, beta, d.ln_eps)  # Eq. 5
        kv = kv.reshape(L, H, dn + dv)
        for h in range(H):
            k = np.concatenate([kv[:, h, :dn], kr], axis=1)
            v = kv[:, h, dn:]
            p = softmax((k @ widen(case.q[b, h], d.dtype)) * softmax_scale(d))
            out[b, h] = p @ v
    return out


# --------------------------------------------------------------------------
# prompt processing (prefill): causal attention over every prompt position
# --------------------------------------------------------------------------
def prefill_latents(pc, b: int):
    """(c~ [L, d_c], k^R [L, d_r]) of prompt b: its packed rows, gated as the
    decode path gates cached rows (Eq. 5 in latent space, or the ablations)."""
    d = pc.dims
    s0, s1 = int(pc.cu_seqlens[b]), int(pc.cu_seqlens[b + 1])
    c = widen(pc.c[s0:s1], d.dtype)
    kr = widen(pc.kr[s0:s1], d.dtype)
    if d.gate and s1 > s0:
        g = widen(pc.gate_table, d.dtype)[pc.ids[s0:s1].astype(np.int64)]
        c = gate_latents(c, g, np.asarray(pc.ln_gamma, np.float64), np.asarray(pc.ln_beta, np.float64),
                         d.ln_eps, getattr(d, "gate_op", "mul_ln"))
    return c, kr


def future_positions(L: int) -> np.ndarray:
    """[L, L] mask of the (query t, key j) pairs with j > t: the keys a query
    of a prompt does not see (the sum of Eq. 13 stops at the query's own
    position, which it includes)."""
    return np.triu(np.ones((L, L), dtype=bool), k=1)


def prefill(pc, batches: Optional[Iterable[int]] = None, heads: Optional[Iterable[int]] = None) -> np.ndarray:
    """u_{t,i} = sum_{j <= t} softmax_j(q_{t,i} . k_{j,i} / sqrt(d_h + d_h^R)) v_{j,i}
    for every position t of every prompt (Eq. 13, whose sum runs over the
    positions up to the query's own), with k_{j,i} = [W_UK,i c~_j ; k^R_j] and
    v_{j,i} = W_UV,i c~_j (Eqs. 2, 6, 12) up-projected from the gated latent:
    the unabsorbed per-head form of the Appendix E listing applied to a whole
    prompt at once, the causal mask written as a full score matrix with the
    entries above the diagonal removed.  Returns [T, H, d_v] float64 (rows of
    unselected prompts or heads NaN)."""
    d = pc.dims
    T, H = pc.total_tokens, d.num_heads
    out = np.full((T, H, d.d_v), np.nan)
    bs = range(pc.batch) if batches is None else list(batches)
    hs = range(H) if heads is None else list(heads)
    for b in bs:
        s0, s1 = int(pc.cu_seqlens[b]), int(pc.cu_seqlens[b + 1])
        L = s1 - s0
        if L == 0:
            continue
        c_t, kr = prefill_latents(pc, b)
        future = future_positions(L)
        for h in hs:
            k = np.concatenate([c_t @ widen(pc.w_uk[h], d.dtype).T, kr], axis=1)   # [L, d_n + d_r]
            v = c_t @ widen(pc.w_uv[h], d.dtype).T                                   # [L, d_v]
            q = widen(pc.q[s0:s1, h], d.dtype)                                      # [L, d_n + d_r]
            s = (q @ k.T) * softmax_scale(d)
            s[future] = -np.inf
            out[s0:s1, h] = softmax(s) @ v
    return out


def prefill_pools(pc):
    """The paged cache after the prompts are written into it: token t of
    prompt b goes to logical position t through the block table (the decode
    steps that follow read it there).  Returns new arrays."""
    c_pool, kr_pool, id_pool = pc.c_pool.copy(), pc.kr_pool.copy(), pc.id_pool.copy()
    P = pc.dims.page_size
    for b in range(pc.batch):
        s0, s1 = int(pc.cu_seqlens[b]), int(pc.cu_seqlens[b + 1])
        for t in range(s1 - s0):
            page, slot = paged_position(pc.block_table, b, t, P)
            c_pool[page, slot] = pc.c[s0 + t]
            kr_pool[page, slot] = pc.kr[s0 + t]
            id_pool[page, slot] = pc.ids[s0 + t]
    return c_pool, kr_pool, id_pool


# --------------------------------------------------------------------------
# one decode step through a whole attention layer (Appendix C, Appendix E)
# --------------------------------------------------------------------------
def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """The bf16 value a model of dtype bf16 stores for x: float64 -> float32 ->
    bf16, each step rounded to nearest, ties to even (NaN kept as a quiet NaN)."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float64).astype(np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    nan = np.isnan(f)
    if nan.any():
        r[nan] = np.uint16(0x7FC0)
    return r


def store(x: np.ndarray, dtype: str) -> np.ndarray:
    """A float64 result kept in the model dtype (bf16 bits, or float64 for fp32
    workloads, whose values the oracle keeps exactly)."""
    return to_bf16_bits(x) if dtype == "bf16" else np.asarray(x, dtype=np.float64)


def rope(x: np.ndarray, pos, theta: float) -> np.ndarray:
    """Rotary position embedding as the listing applies it (apply_rotary_emb with
    freqs_cis): consecutive pairs (x_2i, x_2i+1) of the last axis rotated by the
    angle pos * theta^(-2i/d).  ``pos`` broadcasts against x.shape[:-1]."""
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    freq = theta ** (-2.0 * np.arange(d // 2) / d)
    ang = np.asarray(pos, dtype=np.float64)[..., None] * freq
    c, s = np.cos(ang), np.sin(ang)
    x0, x1 = x[..., 0::2], x[..., 1::2]
    out = np.empty(np.broadcast_shapes(x.shape, ang.shape[:-1] + (d,)), dtype=np.float64)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def rms_norm(x: np.ndarray, w: np.ndarray, eps: float) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * w over the last axis (the listing's kv_norm)."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt((x * x).mean(axis=-1, keepdims=True) + eps) * np.asarray(w, dtype=np.float64)


def layer_step(lc, kv_from=None):
    """The decode-step inputs of the attention (Appendix C with q-LoRA rank 0, as
    every model of Appendix A): q = W^Q x split per head into [q^C ; q^R] with
    q^R rotated (Eqs. 8-9), [c^KV ; k^R] = W^{DKV,KR} x (Eqs. 1 and 10) with k^R
    rotated and c^KV passed through the listing's kv_norm (RMSNorm) before it is
    cached.  The rotation position of a sequence's new token is L_b - 1.
    Returns the decode case of this step: the cache plus (q, c_new, kr_new) as
    the model stores them.

    kv_from: for a later layer of a layer group (Section 5 inter-layer sharing,
    Appendix H), the group's first layer: the group shares W^{DKV,KR} and its
    activations, so this step's c^KV, k^R and id are that layer's and only q is
    this layer's own (its cache, gate table and up-projections are lc.case's)."""
    case = lc.case
    d = case.dims
    H, dn, dr, dc = d.num_heads, d.d_nope, d.d_rope, d.d_c
    B = case.batch
    pos = case.positions().astype(np.float64)
    x = widen(lc.x, d.dtype)
    q = (x @ widen(lc.w_q, d.dtype).T).reshape(B, H, dn + dr)
    q[..., dn:] = rope(q[..., dn:], pos[:, None], lc.rope_theta)
    kv = x @ widen(lc.w_kv_a, d.dtype).T
    c = rms_norm(kv[:, :dc], widen(lc.kv_norm_w, d.dtype), lc.rms_eps)
    kr = rope(kv[:, dc:], pos, lc.rope_theta)
    if kv_from is not None:
        first = layer_step(kv_from)
        return dataclasses.replace(case, q=store(q, d.dtype), c_new=first.c_new, kr_new=first.kr_new,
                                   ids_new=first.ids_new)
    return dataclasses.replace(case, q=store(q, d.dtype), c_new=store(c, d.dtype), kr_new=store(kr, d.dtype))


def layer_decode(lc, batches: Optional[Iterable[int]] = None, kv_from=None) -> np.ndarray:
    """o_t = W^O [u_t,1 ; ... ; u_t,n_h] (Eq. 14) with u the attention output of
    ``decode_unabsorbed`` over the cache after this step's append, kept in the
    model dtype as the layer stores it.  Returns [B, E] float64 (rows of
    unselected batches NaN).  kv_from: as for layer_step."""
    step = layer_step(lc, kv_from)
    d = step.dims
    u = decode_unabsorbed(step, batches=batches)
    B = step.batch
    y = np.full((B, lc.n_embd), np.nan)
    bs = range(B) if batches is None else list(batches)
    w_o = widen(lc.w_o, d.dtype)
    for b in bs:
        y[b] = w_o @ widen(store(u[b], d.dtype), d.dtype).reshape(-1)
    return y


# --------------------------------------------------------------------------
# cache size (Table 5 and the Appendix F table)
# --------------------------------------------------------------------------
def kv_elements_per_token(kind: str, n_layers: int, *, n_heads: int = 0, d_head: int = 0,
                          n_groups: int = 0, d_c: int = 0, d_rope: int = 0, r: int = 1) -> int:
    """KV-cache elements stored per token over all layers (Table 5).

    mha: 2 n_h d_h l;  gqa: 2 n_g d_h l;  mqa: 2 d_h l;  mla: (d_c + d_h^R) l;
    egmla: (d_c / r + d_h^R) l  (d_c / r is the latent width the cache actually keeps)."""
    if kind == "mha":
        return 2 * n_heads * d_head * n_layers
    if kind == "gqa":
        return 2 * n_groups * d_head * n_layers
    if kind == "mqa":
        return 2 * d_head * n_layers
    if kind == "mla":
        return (d_c + d_rope) * n_layers
    if kind == "egmla":
        if d_c % r:
            raise ValueError("d_c must be divisible by r")
        return (d_c // r + d_rope) * n_layers
    raise ValueError(kind)


def kv_bytes_per_token(d_c: int, d_rope: int, n_layers: int, elem_bytes: int,
                       with_token_id: bool) -> int:
    """Bytes the paged cache keeps per token: (d_c + d_r) values per layer, plus the
    4-byte token id per layer that read-time gating needs to find g = G[id]."""
    return n_layers * ((d_c + d_rope) * elem_bytes + (4 if with_token_id else 0))


def embedding_params(n_layers: int, vocab: int, d_e: int) -> int:
    """Per-layer gate embedding tables: l * V * d_e parameters (Appendix A 'Embed Size')."""
    return n_layers * vocab * d_e

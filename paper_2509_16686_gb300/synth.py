"""Seeded synthetic inputs for EG-MLA decode, shared by the tests, the bench and
the oracle's tests.

This module only draws random numbers and lays them out in the storage formats
the library consumes (paged latent cache, block tables, bf16 bit patterns).  It
holds none of the method's arithmetic: no gating, normalisation or attention.

Workloads mirror the paper's models (Appendix A hyper-parameter table: RoPE dim
64, nope head dim = value head dim, q_lora_rank 0) at five sizes:

  tiny   fp32  B=1   H=4  d_n=32  d_r=16 d_c=64  L=128        V=1000
  c4k    bf16  B=32  H=16 d_n=128 d_r=64 d_c=256 L=4096       V=32000 contiguous pages
  c32k   bf16  B=8   H=16 d_n=128 d_r=64 d_c=256 L=32768      V=32000 permuted shared pool
  ragged bf16  B=128 H=16 d_n=128 d_r=64 d_c=192 L~logU[128,16384] V=50000 Zipf(1.1) ids
  layers bf16  24 layers, B=64 H=16 d_c=256 L=8192 V=50000 (one pool and gate table per layer)

Value distributions: latents N(0,1) (x0.5 for the bf16 workloads), RoPE keys and
queries N(0,1), gate table N(1, 0.1), W_UK / W_UV N(0, d_c^-1/2), LayerNorm
gamma=1, beta=0 unless ``affine_ln`` asks for gamma~N(1,0.1), beta~N(0,0.1).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

PAGE_SIZE = 64
BF16_NAN = np.uint16(0x7FC0)


# --------------------------------------------------------------------------
# storage helpers (bit-level, no arithmetic of the method)
# --------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (round-to-nearest-even), returned as uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bfloat16 bit patterns to float32."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


@dataclasses.dataclass
class Dims:
    num_heads: int
    d_nope: int
    d_rope: int
    d_v: int
    d_c: int
    page_size: int
    vocab: int
    dtype: str          # "bf16" | "fp32"
    gate: bool = True   # False: plain MLA (gate and LayerNorm off)
    # with the gate on: "mul_ln" c~ = LN(c (*) g) (the method), or the paper's
    # ablations "mul" (LayerNorm removed) and "add_ln" ((*) replaced by +)
    gate_op: str = "mul_ln"
    ln_eps: float = 1e-5
    softmax_scale: float = 0.0   # <= 0: the method's default scale (the consumer's rule)


@dataclasses.dataclass
class Case:
    """One decode step's inputs.

    Arrays of the model dtype are stored as uint16 bf16 bits ("bf16") or
    float32 ("fp32").  ``c_pool``/``kr_pool``/``id_pool`` already hold the first
    ``seq_lens[b]-1`` tokens of every sequence; the new token (``c_new`` ...) is
    appended at logical position ``seq_lens[b]-1`` before attention.
    Unused cache slots hold NaN latents and out-of-range ids so that any read of
    them shows up in the result.
    """
    name: str
    dims: Dims
    seed: int
    c_pool: np.ndarray        # [num_pages, P, d_c]
    kr_pool: np.ndarray       # [num_pages, P, d_r]
    id_pool: np.ndarray       # [num_pages, P] int32
    block_table: np.ndarray   # [B, max_pages] int32
    seq_lens: np.ndarray      # [B] int32, includes the new token
    c_new: np.ndarray         # [B, d_c]
    kr_new: np.ndarray        # [B, d_r]
    ids_new: np.ndarray       # [B] int32
    q: np.ndarray             # [B, H, d_nope + d_rope], RoPE already applied
    gate_table: np.ndarray    # [V, d_c]
    ln_gamma: np.ndarray      # [d_c] float32
    ln_beta: np.ndarray       # [d_c] float32
    w_uk: np.ndarray          # [H, d_nope, d_c]
    w_uv: np.ndarray          # [H, d_v, d_c]
    logical_c: Optional[list] = None     # per sequence [L_b, d_c] (after append)
    logical_kr: Optional[list] = None
    logical_ids: Optional[list] = None

    @property
    def batch(self) -> int:
        return int(self.seq_lens.shape[0])

    @property
    def num_pages(self) -> int:
        return int(self.c_pool.shape[0])

    @property
    def max_pages(self) -> int:
        return int(self.block_table.shape[1])

    def positions(self) -> np.ndarray:
        return (self.seq_lens - 1).astype(np.int32)


def _normal(rng: np.random.Generator, shape, std: float, mean: float = 0.0) -> np.ndarray:
    x = rng.standard_normal(size=shape, dtype=np.float32)
    if std != 1.0:
        x *= np.float32(std)
    if mean != 0.0:
        x += np.float32(mean)
    return x


def _store(x: np.ndarray, dtype: str) -> np.ndarray:
    return f32_to_bf16_bits(x) if dtype == "bf16" else np.ascontiguousarray(x, np.float32)


def _nan_fill(dtype: str):
    return BF16_NAN if dtype == "bf16" else np.float32(np.nan)


def zipf_ids(rng: np.random.Generator, n: int, vocab: int, a: float = 1.1) -> np.ndarray:
    """Token ids with Zipf(a) ranks; ranks above the vocabulary are redrawn; id = rank-1."""
    out = np.empty(n, dtype=np.int64)
    filled = 0
    while filled < n:
        r = rng.zipf(a, size=max(2 * (n - filled), 1024))
        r = r[r <= vocab]
        take = min(r.size, n - filled)
        out[filled:filled + take] = r[:take]
        filled += take
    return (out - 1).astype(np.int32)


def log_uniform_lengths(rng: np.random.Generator, n: int, lo: int, hi: int) -> np.ndarray:
    """L = floor(exp(U[ln lo, ln hi])), clamped to [lo, hi]."""
    u = rng.uniform(math.log(lo), math.log(hi), size=n)
    return np.clip(np.floor(np.exp(u)), lo, hi).astype(np.int32)


def make_case(name: str, dims: Dims, seq_lens, *, seed: int, latent_scale: float = 1.0,
              id_dist: str = "uniform", layout: str = "contiguous", affine_ln: bool = False,
              keep_logical: bool = True, extra_pages: int = 0) -> Case:
    """Build one synthetic decode step.

    layout: "contiguous" (sequence b owns pages [b*maxP, ...)), "permuted" (the
    pages every sequence needs are shuffled over one shared pool) or
    "shuffled_pool" (permuted, plus ``extra_pages`` unused pages in the pool).
    """
    rng = np.random.default_rng(seed)
    P = dims.page_size
    seq_lens = np.asarray(seq_lens, dtype=np.int32)
    B = seq_lens.shape[0]
    npg = [(int(L) + P - 1) // P for L in seq_lens]
    max_pages = max(max(npg), 1)
    if layout == "contiguous":
        num_pages = B * max_pages
        block_table = np.zeros((B, max_pages), dtype=np.int32)
        for b in range(B):
            block_table[b, :] = b * max_pages + np.arange(max_pages, dtype=np.int32)
    else:
        need = int(sum(npg))
        num_pages = need + int(extra_pages)
        perm = rng.permutation(num_pages).astype(np.int32)
        block_table = np.zeros((B, max_pages), dtype=np.int32)
        k = 0
        for b in range(B):
            block_table[b, :npg[b]] = perm[k:k + npg[b]]
            k += npg[b]
            # slots past the sequence point at a valid but unrelated page
            if npg[b] < max_pages:
                block_table[b, npg[b]:] = perm[-1]
    num_pages = max(num_pages, 1)

    dt = dims.dtype
    H, dn, dr, dv, dc, V = dims.num_heads, dims.d_nope, dims.d_rope, dims.d_v, dims.d_c, dims.vocab
    c_pool = np.full((num_pages, P, dc), _nan_fill(dt), dtype=np.uint16 if dt == "bf16" else np.float32)
    kr_pool = np.full((num_pages, P, dr), _nan_fill(dt), dtype=c_pool.dtype)
    id_pool = np.full((num_pages, P), -7, dtype=np.int32)

    logical_c, logical_kr, logical_ids = [], [], []
    for b in range(B):
        L = int(seq_lens[b])
        c = _store(_normal(rng, (L, dc), latent_scale), dt)
        kr = _store(_normal(rng, (L, dr), 1.0), dt)
        if id_dist == "zipf":
            ids = zipf_ids(rng, L, V)
        else:
            ids = rng.integers(0, V, size=L, dtype=np.int64).astype(np.int32)
        if keep_logical:
            logical_c.append(c)
            logical_kr.append(kr)
            logical_ids.append(ids)
        # the first L-1 tokens are already cached; the last one is appended
        for j in range(0, L - 1, P):
            n = min(P, L - 1 - j)
            page = block_table[b, j // P]
            c_pool[page, :n] = c[j:j + n]
            kr_pool[page, :n] = kr[j:j + n]
            id_pool[page, :n] = ids[j:j + n]
        if b == 0:
            c_new = np.zeros((B, dc), dtype=c.dtype)
            kr_new = np.zeros((B, dr), dtype=kr.dtype)
            ids_new = np.zeros((B,), dtype=np.int32)
        if L > 0:
            c_new[b] = c[L - 1]
            kr_new[b] = kr[L - 1]
            ids_new[b] = ids[L - 1]

    q = _store(_normal(rng, (B, H, dn + dr), 1.0), dt)
    gate_table = _store(_normal(rng, (V, dc), 0.1, mean=1.0), dt)
    wstd = dc ** -0.5   # std of the N(0, d_c^-1/2) draw
    w_uk = _store(_normal(rng, (H, dn, dc), wstd), dt)
    w_uv = _store(_normal(rng, (H, dv, dc), wstd), dt)
    if affine_ln:
        ln_gamma = _normal(rng, (dc,), 0.1, mean=1.0)
        ln_beta = _normal(rng, (dc,), 0.1)
    else:
        ln_gamma = np.ones((dc,), dtype=np.float32)
        ln_beta = np.zeros((dc,), dtype=np.float32)
    return Case(name=name, dims=dims, seed=seed, c_pool=c_pool, kr_pool=kr_pool, id_pool=id_pool,
                block_table=block_table, seq_lens=seq_lens, c_new=c_new, kr_new=kr_new,
                ids_new=ids_new, q=q, gate_table=gate_table, ln_gamma=ln_gamma, ln_beta=ln_beta,
                w_uk=w_uk, w_uv=w_uv,
                logical_c=logical_c if keep_logical else None,
                logical_kr=logical_kr if keep_logical else None,
                logical_ids=logical_ids if keep_logical else None)


# --------------------------------------------------------------------------
# the five workloads
# --------------------------------------------------------------------------
def dims_tiny() -> Dims:
    return Dims(num_heads=4, d_nope=32, d_rope=16, d_v=32, d_c=64, page_size=PAGE_SIZE,
                vocab=1000, dtype="fp32")


def dims_bf16(d_c: int = 256, vocab: int = 32000, gate: bool = True, gate_op: str = "mul_ln") -> Dims:
    return Dims(num_heads=16, d_nope=128, d_rope=64, d_v=128, d_c=d_c, page_size=PAGE_SIZE,
                vocab=vocab, dtype="bf16", gate=gate, gate_op=gate_op)


def case_tiny(seed: int = 0, **kw) -> Case:
    """fp32, batch 1, 4 heads, 32+16 head dim, d_c 64, context 128, vocab 1000."""
    return make_case("tiny", dims_tiny(), [128], seed=seed, **kw)


def case_c4k(seed: int = 1, batch: int = 32, ctx: int = 4096, **kw) -> Case:
    """bf16, batch 32, 16 heads, d_c 256, context 4096, contiguous 64-token pages."""
    return make_case("c4k", dims_bf16(), [ctx] * batch, seed=seed, latent_scale=0.5, **kw)


def case_c32k(seed: int = 2, batch: int = 8, ctx: int = 32768, **kw) -> Case:
    """bf16, batch 8, context 32768, block table permuted over a shared page pool."""
    kw.setdefault("layout", "permuted")
    return make_case("c32k", dims_bf16(), [ctx] * batch, seed=seed, latent_scale=0.5, **kw)


def ragged_lengths(seed: int = 3, batch: int = 128, lo: int = 128, hi: int = 16384) -> np.ndarray:
    return log_uniform_lengths(np.random.default_rng(seed + 1000), batch, lo, hi)


def case_ragged(seed: int = 3, batch: int = 128, gate: bool = True, **kw) -> Case:
    """bf16, batch 128, log-uniform contexts in [128, 16384], d_c 192, Zipf(1.1) ids.

    With ``gate=False`` this is the plain-MLA baseline at d_c 512 on the same lengths.
    """
    lens = ragged_lengths(seed, batch)
    d_c = 192 if gate else 512
    kw.setdefault("layout", "permuted")
    return make_case("ragged" if gate else "ragged_mla", dims_bf16(d_c=d_c, vocab=50000, gate=gate),
                     lens, seed=seed, latent_scale=0.5, id_dist="zipf", **kw)


def case_layer(layer: int, seed: int = 4, batch: int = 64, ctx: int = 8192, **kw) -> Case:
    """One attention layer of the 24-layer decoder step (hidden 2048, 16 heads, d_c 256)."""
    kw.setdefault("keep_logical", False)
    return make_case(f"layers[{layer}]", dims_bf16(vocab=50000), [ctx] * batch,
                     seed=seed * 1000 + layer, latent_scale=0.5, **kw)


N_LAYERS = 24


# --------------------------------------------------------------------------
# one full attention layer of a decode step
# --------------------------------------------------------------------------
F32_EPS = float(np.finfo(np.float32).eps)


@dataclasses.dataclass
class LayerCase:
    """Inputs of one decode step through a whole EG-MLA attention layer.

    ``case`` holds the cache (its first ``seq_lens[b]-1`` tokens), the gate
    table, LayerNorm and absorbed weights; its ``q``/``c_new``/``kr_new`` are
    not used: the layer derives them from the hidden state ``x``.  Weights have
    the PyTorch Linear layout [out, in] in the model dtype.
    """
    case: Case
    n_embd: int
    x: np.ndarray           # [B, E]
    w_q: np.ndarray         # [H (d_nope + d_rope), E]
    w_kv_a: np.ndarray      # [d_c + d_rope, E]
    kv_norm_w: np.ndarray   # [d_c]
    w_o: np.ndarray         # [E, H d_v]
    rope_theta: float = 10000.0
    rms_eps: float = F32_EPS


@dataclasses.dataclass
class R0Inputs:
    """The extra inputs of the paper-literal (R0) gate placement: the joint
    up-projection W^UKV (per head its key rows W_UK,h, then its value rows
    W_UV,h: the case's own weights in the row order of Appendix E), a gate
    table in that H (d_n + d_v)-wide space, and its LayerNorm's gamma, beta."""
    w_ukv: np.ndarray      # [H (d_n + d_v), d_c] model dtype bits
    gate_r0: np.ndarray    # [V, H (d_n + d_v)] model dtype bits
    gamma: np.ndarray      # [H (d_n + d_v)] float32
    beta: np.ndarray       # [H (d_n + d_v)] float32


def make_r0_inputs(case: Case, *, seed: int, affine: bool = True) -> R0Inputs:
    """Seeded R0 inputs for `case`: gate table N(1, 0.1) like the latent gate
    table, gamma N(1, 0.1) and beta N(0, 0.1) (or 1 and 0)."""
    d = case.dims
    rng = np.random.default_rng(seed)
    width = d.num_heads * (d.d_nope + d.d_v)
    w_ukv = np.concatenate([case.w_uk, case.w_uv], axis=1).reshape(width, d.d_c)
    gate = _store(_normal(rng, (d.vocab, width), 0.1, mean=1.0), d.dtype)
    gamma = _normal(rng, (width,), 0.1, mean=1.0) if affine else np.ones(width, np.float32)
    beta = _normal(rng, (width,), 0.1) if affine else np.zeros(width, np.float32)
    return R0Inputs(w_ukv=np.ascontiguousarray(w_ukv), gate_r0=gate, gamma=np.asarray(gamma, np.float32),
                    beta=np.asarray(beta, np.float32))


def make_layer_case(case: Case, n_embd: int, *, seed: int, rope_theta: float = 10000.0,
                    rms_eps: float = F32_EPS) -> LayerCase:
    """Hidden state N(0, 1) and projection weights N(0, fan_in^-1/2); the
    RMSNorm weight N(1, 0.1)."""
    rng = np.random.default_rng(seed)
    d, dt = case.dims, case.dims.dtype
    H, dn, dr, dv, dc, E = d.num_heads, d.d_nope, d.d_rope, d.d_v, d.d_c, n_embd
    B = case.batch
    return LayerCase(
        case=case, n_embd=E,
        x=_store(_normal(rng, (B, E), 1.0), dt),
        w_q=_store(_normal(rng, (H * (dn + dr), E), E ** -0.5), dt),
        w_kv_a=_store(_normal(rng, (dc + dr, E), E ** -0.5), dt),
        kv_norm_w=_store(_normal(rng, (dc,), 0.1, mean=1.0), dt),
        w_o=_store(_normal(rng, (E, H * dv), (H * dv) ** -0.5), dt),
        rope_theta=rope_theta, rms_eps=rms_eps)


# --------------------------------------------------------------------------
# prompt processing (prefill): prompts packed one after another
# --------------------------------------------------------------------------
@dataclasses.dataclass
class PrefillCase:
    """One prefill call: B prompts packed token after token (prompt b holds
    rows ``cu_seqlens[b] .. cu_seqlens[b+1]-1`` of every per-token array), the
    layer's gate table, LayerNorm and up-projections, and an empty paged cache
    (NaN latents, out-of-range ids) that the call fills with the prompts.
    Arrays of the model dtype are stored as in ``Case``."""
    name: str
    dims: Dims
    seed: int
    seq_lens: np.ndarray      # [B] int32
    cu_seqlens: np.ndarray    # [B + 1] int32
    q: np.ndarray             # [T, H, d_nope + d_rope], RoPE already applied
    c: np.ndarray             # [T, d_c]
    kr: np.ndarray            # [T, d_r]
    ids: np.ndarray           # [T] int32
    gate_table: np.ndarray    # [V, d_c]
    ln_gamma: np.ndarray      # [d_c] float32
    ln_beta: np.ndarray       # [d_c] float32
    w_uk: np.ndarray          # [H, d_nope, d_c]
    w_uv: np.ndarray          # [H, d_v, d_c]
    c_pool: np.ndarray        # [num_pages, P, d_c]
    kr_pool: np.ndarray       # [num_pages, P, d_r]
    id_pool: np.ndarray       # [num_pages, P] int32
    block_table: np.ndarray   # [B, max_pages] int32

    @property
    def batch(self) -> int:
        return int(self.seq_lens.shape[0])

    @property
    def total_tokens(self) -> int:
        return int(self.cu_seqlens[-1])

    @property
    def num_pages(self) -> int:
        return int(self.c_pool.shape[0])

    @property
    def max_pages(self) -> int:
        return int(self.block_table.shape[1])


def make_prefill_case(name: str, dims: Dims, seq_lens, *, seed: int, latent_scale: float = 0.5,
                      id_dist: str = "uniform", affine_ln: bool = False, extra_pages: int = 0,
                      q_zero: bool = False) -> PrefillCase:
    """Seeded prompts with the value distributions of the decode workloads; the
    cache pages of all prompts are shuffled over one pool (plus ``extra_pages``
    unused ones)."""
    rng = np.random.default_rng(seed)
    P = dims.page_size
    seq_lens = np.asarray(seq_lens, dtype=np.int32)
    B = seq_lens.shape[0]
    cu = np.zeros(B + 1, dtype=np.int32)
    cu[1:] = np.cumsum(seq_lens)
    T = int(cu[-1])
    npg = [(int(L) + P - 1) // P for L in seq_lens]
    max_pages = max(max(npg) if npg else 1, 1)
    num_pages = max(int(sum(npg)) + int(extra_pages), 1)
    perm = rng.permutation(num_pages).astype(np.int32)
    block_table = np.full((B, max_pages), perm[-1], dtype=np.int32)
    k = 0
    for b in range(B):
        block_table[b, :npg[b]] = perm[k:k + npg[b]]
        k += npg[b]

    dt = dims.dtype
    H, dn, dr, dv, dc, V = dims.num_heads, dims.d_nope, dims.d_rope, dims.d_v, dims.d_c, dims.vocab
    c = _store(_normal(rng, (T, dc), latent_scale), dt)
    kr = _store(_normal(rng, (T, dr), 1.0), dt)
    ids = zipf_ids(rng, T, V) if id_dist == "zipf" else rng.integers(0, V, size=T, dtype=np.int64).astype(np.int32)
    q = _normal(rng, (T, H, dn + dr), 1.0)
    if q_zero:
        q[:] = 0.0
    q = _store(q, dt)
    gate_table = _store(_normal(rng, (V, dc), 0.1, mean=1.0), dt)
    wstd = dc ** -0.5
    w_uk = _store(_normal(rng, (H, dn, dc), wstd), dt)
    w_uv = _store(_normal(rng, (H, dv, dc), wstd), dt)
    if affine_ln:
        ln_gamma = _normal(rng, (dc,), 0.1, mean=1.0)
        ln_beta = _normal(rng, (dc,), 0.1)
    else:
        ln_gamma = np.ones((dc,), dtype=np.float32)
        ln_beta = np.zeros((dc,), dtype=np.float32)
    c_pool = np.full((num_pages, P, dc), _nan_fill(dt), dtype=np.uint16 if dt == "bf16" else np.float32)
    kr_pool = np.full((num_pages, P, dr), _nan_fill(dt), dtype=c_pool.dtype)
    id_pool = np.full((num_pages, P), -7, dtype=np.int32)
    return PrefillCase(name=name, dims=dims, seed=seed, seq_lens=seq_lens, cu_seqlens=cu, q=q, c=c, kr=kr,
                       ids=ids.astype(np.int32), gate_table=gate_table, ln_gamma=np.asarray(ln_gamma, np.float32),
                       ln_beta=np.asarray(ln_beta, np.float32), w_uk=w_uk, w_uv=w_uv, c_pool=c_pool,
                       kr_pool=kr_pool, id_pool=id_pool, block_table=block_table)


def case_prefill(seed: int = 5, batch: int = 8, prompt: int = 4096, **kw) -> PrefillCase:
    """bf16, 8 prompts of 4096 tokens, 16 heads, d_c 256, vocab 32000 (the
    shapes of the 4K decode workload)."""
    return make_prefill_case("prefill", dims_bf16(), [prompt] * batch, seed=seed, **kw)


def case_prefill_ragged(seed: int = 6, batch: int = 16, lo: int = 128, hi: int = 4096, **kw) -> PrefillCase:
    """bf16, 16 prompts with log-uniform lengths in [128, 4096], d_c 192,
    vocab 50000, Zipf(1.1) ids (the shapes of the ragged decode workload)."""
    lens = log_uniform_lengths(np.random.default_rng(seed + 1000), batch, lo, hi)
    kw.setdefault("id_dist", "zipf")
    return make_prefill_case("prefill_ragged", dims_bf16(d_c=192, vocab=50000), lens, seed=seed, **kw)


def make_embedding(case, d_e: int, *, seed: int):
    """Gate embedding of the non-precomputed EG-MLA form (Section 3 Eqs. 3-4):
    E [V, d_e] ~ N(0, 1) and W^UE [d_c, d_e] ~ N(0, d_e^-1/2), stored in the
    model dtype, so that E W^UE^T has unit-variance entries."""
    d = case.dims
    rng = np.random.default_rng(seed)
    emb = _store(_normal(rng, (d.vocab, d_e), 1.0), d.dtype)
    w_ue = _store(_normal(rng, (d.d_c, d_e), d_e ** -0.5), d.dtype)
    return emb, w_ue

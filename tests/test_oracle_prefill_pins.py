"""Pins of the oracle's prefill (every position of a prompt at once) against
things other than itself: the pinned decode oracle on each prefix, torch's
causal scaled_dot_product_attention, closed forms and invariants.  CPU only."""
from __future__ import annotations

import dataclasses

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import egmla_oracle as orc
from paper_2509_16686_gb300 import synth


def small_prefill(seed=0, lens=(1, 19, 40, 0, 33), H=3, dn=8, dr=4, dv=8, dc=16, V=50, P=16,
                  affine=True, gate=True, gate_op="mul_ln", dtype="fp32", q_zero=False):
    dims = synth.Dims(num_heads=H, d_nope=dn, d_rope=dr, d_v=dv, d_c=dc, page_size=P, vocab=V,
                      dtype=dtype, gate=gate, gate_op=gate_op)
    return synth.make_prefill_case("small_prefill", dims, list(lens), seed=seed, affine_ln=affine,
                                   extra_pages=2, latent_scale=1.0, q_zero=q_zero)


def rel_err(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def prefix_decode_case(pc, b: int, t: int) -> synth.Case:
    """The decode step of query t of prompt b over the prompt's first t + 1
    tokens: the cache the prefill wrote, the new token = token t."""
    c_pool, kr_pool, id_pool = orc.prefill_pools(pc)
    r = int(pc.cu_seqlens[b]) + t
    return synth.Case(name="prefix", dims=pc.dims, seed=pc.seed, c_pool=c_pool, kr_pool=kr_pool,
                      id_pool=id_pool, block_table=pc.block_table[b:b + 1].copy(),
                      seq_lens=np.array([t + 1], np.int32), c_new=pc.c[r:r + 1].copy(),
                      kr_new=pc.kr[r:r + 1].copy(), ids_new=pc.ids[r:r + 1].copy(),
                      q=pc.q[r:r + 1].copy(), gate_table=pc.gate_table, ln_gamma=pc.ln_gamma,
                      ln_beta=pc.ln_beta, w_uk=pc.w_uk, w_uv=pc.w_uv)


def torch_gated(pc, b):
    """c~ of prompt b through torch's layer_norm (library routine)."""
    d = pc.dims
    s0, s1 = int(pc.cu_seqlens[b]), int(pc.cu_seqlens[b + 1])
    c = torch.from_numpy(orc.widen(pc.c[s0:s1], d.dtype))
    if not d.gate:
        return c
    g = torch.from_numpy(orc.widen(pc.gate_table, d.dtype))[torch.from_numpy(pc.ids[s0:s1].astype(np.int64))]
    return F.layer_norm(c * g, (d.d_c,), weight=torch.from_numpy(pc.ln_gamma.astype(np.float64)),
                        bias=torch.from_numpy(pc.ln_beta.astype(np.float64)), eps=d.ln_eps)


# --------------------------------------------------------------------------- row t = decode of the prefix
@pytest.mark.parametrize("gate_op", ["mul_ln", "mul", "add_ln"])
def test_prefill_rows_equal_decode_of_the_prefix(gate_op):
    pc = small_prefill(gate_op=gate_op)
    got = orc.prefill(pc)
    for b in range(pc.batch):
        L = int(pc.seq_lens[b])
        for t in range(L):
            want = orc.decode_unabsorbed(prefix_decode_case(pc, b, t))[0]
            row = got[int(pc.cu_seqlens[b]) + t]
            assert rel_err(row, want) < 1e-12, (b, t)


def test_prefill_rows_equal_decode_gate_off_bf16():
    pc = small_prefill(gate=False, dtype="bf16", seed=3)
    got = orc.prefill(pc)
    for b in range(pc.batch):
        for t in range(0, int(pc.seq_lens[b]), 5):
            want = orc.decode_unabsorbed(prefix_decode_case(pc, b, t))[0]
            assert rel_err(got[int(pc.cu_seqlens[b]) + t], want) < 1e-12


# --------------------------------------------------------------------------- library routine
@pytest.mark.parametrize("gate", [True, False])
def test_prefill_matches_torch_causal_sdpa_with_identity_projections(gate):
    """d_c = d_n = d_v and W_UK,h = W_UV,h = I: keys [c~ ; k^R], values c~, so
    every head is torch's causal scaled_dot_product_attention on those."""
    pc = small_prefill(dn=16, dv=16, dc=16, gate=gate, seed=5)
    eye = np.broadcast_to(np.eye(16, dtype=np.float32), (pc.dims.num_heads, 16, 16)).copy()
    pc = dataclasses.replace(pc, w_uk=eye, w_uv=eye.copy())
    got = orc.prefill(pc)
    d = pc.dims
    for b in range(pc.batch):
        s0, s1 = int(pc.cu_seqlens[b]), int(pc.cu_seqlens[b + 1])
        if s1 == s0:
            continue
        c = torch_gated(pc, b)
        kr = torch.from_numpy(orc.widen(pc.kr[s0:s1], d.dtype))
        k = torch.cat([c, kr], dim=-1)
        for h in range(d.num_heads):
            q = torch.from_numpy(orc.widen(pc.q[s0:s1, h], d.dtype))
            want = F.scaled_dot_product_attention(q[None], k[None], c[None], is_causal=True)[0].numpy()
            assert rel_err(got[s0:s1, h], want) < 1e-12, (b, h)


# --------------------------------------------------------------------------- closed forms
def test_prefill_single_token_closed_form():
    """A one-token prompt attends only to itself: u = W_UV c~_0."""
    pc = small_prefill(lens=(1, 1, 1), seed=7)
    got = orc.prefill(pc)
    d = pc.dims
    for b in range(pc.batch):
        c = torch_gated(pc, b).numpy()[0]
        for h in range(d.num_heads):
            want = orc.widen(pc.w_uv[h], d.dtype) @ c
            np.testing.assert_allclose(got[b, h], want, rtol=1e-12, atol=1e-13)


def test_prefill_zero_query_is_the_causal_running_mean():
    """q = 0 gives equal weights over the visible keys: u_t = W_UV (1/(t+1)) sum_{j<=t} c~_j."""
    pc = small_prefill(q_zero=True, seed=8)
    got = orc.prefill(pc)
    d = pc.dims
    for b in range(pc.batch):
        s0, s1 = int(pc.cu_seqlens[b]), int(pc.cu_seqlens[b + 1])
        if s1 == s0:
            continue
        c = torch_gated(pc, b).numpy()
        mean = np.cumsum(c, axis=0) / np.arange(1, s1 - s0 + 1)[:, None]
        for h in range(d.num_heads):
            want = mean @ orc.widen(pc.w_uv[h], d.dtype).T
            np.testing.assert_allclose(got[s0:s1, h], want, rtol=1e-11, atol=1e-12)


# --------------------------------------------------------------------------- invariants
def test_prefill_is_causal():
    """Changing the tokens after position t changes no output row up to t."""
    pc = small_prefill(lens=(40,), seed=9)
    base = orc.prefill(pc)
    t = 17
    c = pc.c.copy(); c[t + 1:] = -c[t + 1:] + 0.5
    kr = pc.kr.copy(); kr[t + 1:] *= 3.0
    ids = pc.ids.copy(); ids[t + 1:] = (ids[t + 1:] + 7) % pc.dims.vocab
    q = pc.q.copy(); q[t + 1:] *= -1.0
    got = orc.prefill(dataclasses.replace(pc, c=c, kr=kr, ids=ids, q=q))
    np.testing.assert_array_equal(got[:t + 1], base[:t + 1])
    assert rel_err(got[t + 1:], base[t + 1:]) > 1e-3


def test_prompts_are_independent():
    """A packed batch gives, prompt by prompt, what each prompt gives alone."""
    pc = small_prefill(seed=10)
    got = orc.prefill(pc)
    for b in range(pc.batch):
        s0, s1 = int(pc.cu_seqlens[b]), int(pc.cu_seqlens[b + 1])
        alone = dataclasses.replace(pc, seq_lens=pc.seq_lens[b:b + 1].copy(),
                                    cu_seqlens=np.array([0, s1 - s0], np.int32), q=pc.q[s0:s1],
                                    c=pc.c[s0:s1], kr=pc.kr[s0:s1], ids=pc.ids[s0:s1],
                                    block_table=pc.block_table[b:b + 1])
        np.testing.assert_allclose(orc.prefill(alone), got[s0:s1], rtol=1e-13, atol=1e-14)


def test_prefill_pool_write_is_the_prompt_through_the_block_table():
    pc = small_prefill(seed=11)
    c_pool, kr_pool, id_pool = orc.prefill_pools(pc)
    P = pc.dims.page_size
    written = np.zeros(id_pool.shape, dtype=bool)
    for b in range(pc.batch):
        s0, s1 = int(pc.cu_seqlens[b]), int(pc.cu_seqlens[b + 1])
        np.testing.assert_array_equal(orc.gather_sequence(c_pool, pc.block_table, b, s1 - s0, P), pc.c[s0:s1])
        np.testing.assert_array_equal(orc.gather_sequence(kr_pool, pc.block_table, b, s1 - s0, P), pc.kr[s0:s1])
        np.testing.assert_array_equal(orc.gather_sequence(id_pool, pc.block_table, b, s1 - s0, P), pc.ids[s0:s1])
        for t in range(s1 - s0):
            written[pc.block_table[b, t // P], t % P] = True
    assert np.isnan(c_pool[~written]).all() and np.isnan(kr_pool[~written]).all()
    assert (id_pool[~written] == -7).all()


# --------------------------------------------------------------------------- planted mistakes
@pytest.mark.parametrize("mistake", ["self_excluded", "no_mask", "anti_causal", "reversed_keys"])
def test_prefill_pins_catch_planted_mistakes(mistake, monkeypatch):
    pc = small_prefill(lens=(19, 33), seed=12)
    want = np.stack([orc.decode_unabsorbed(prefix_decode_case(pc, 1, t))[0] for t in range(33)])
    base_sm = orc.softmax
    if mistake == "self_excluded":
        monkeypatch.setattr(orc, "future_positions", lambda L: np.triu(np.ones((L, L), bool), k=0))
    elif mistake == "no_mask":
        monkeypatch.setattr(orc, "future_positions", lambda L: np.zeros((L, L), bool))
    elif mistake == "anti_causal":
        monkeypatch.setattr(orc, "future_positions", lambda L: np.tril(np.ones((L, L), bool), k=-1))
    else:
        monkeypatch.setattr(orc, "softmax", lambda s: base_sm(s[..., ::-1]))
    with np.errstate(invalid="ignore"):
        got = orc.prefill(pc)[19:52]
    assert not np.allclose(got, want, rtol=1e-6, atol=1e-8), mistake

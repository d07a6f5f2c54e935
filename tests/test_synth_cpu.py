"""The seeded input generator draws what the design's input recipe states:
value distributions, token-id and length structure, page layouts, and the NaN
fill of unused cache slots (CPU only)."""
import math

import numpy as np

from paper_2509_16686_gb300 import synth


def f(bits):
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


def test_value_distributions_of_a_bf16_workload():
    case = synth.make_case("recipe", synth.dims_bf16(), [4096] * 4, seed=1, latent_scale=0.5)
    c = np.concatenate([f(x) for x in case.logical_c])
    assert abs(c.mean()) < 0.01 and abs(c.std() - 0.5) < 0.01            # latents N(0, 1) x 0.5
    kr = np.concatenate([f(x) for x in case.logical_kr])
    assert abs(kr.std() - 1.0) < 0.02                                     # RoPE keys N(0, 1)
    g = f(case.gate_table)
    assert abs(g.mean() - 1.0) < 0.002 and abs(g.std() - 0.1) < 0.002    # gate table N(1, 0.1)
    w = f(case.w_uk)
    assert abs(w.std() - 1.0 / math.sqrt(256)) < 0.002                   # W_UK N(0, d_c^-1/2)
    assert (case.ln_gamma == 1).all() and (case.ln_beta == 0).all()


def test_zipf_ids_and_log_uniform_lengths():
    rng = np.random.default_rng(0)
    ids = synth.zipf_ids(rng, 200000, 50000)
    assert ids.min() >= 0 and ids.max() < 50000
    counts = np.bincount(ids, minlength=50000)
    # Zipf(1.1): rank 1 is the most frequent and about 2^1.1 times rank 2
    assert counts.argmax() == 0 and 1.8 < counts[0] / counts[1] < 2.5
    L = synth.log_uniform_lengths(rng, 100000, 128, 16384)
    assert L.min() >= 128 and L.max() <= 16384
    # log-uniform: as many lengths in [128, 1024) as in [2048, 16384)
    a, b = ((L >= 128) & (L < 1024)).mean(), ((L >= 2048) & (L < 16384)).mean()
    assert abs(a - b) < 0.02


def test_page_layouts_and_unused_slots():
    dims = synth.dims_bf16(vocab=1000)
    cont = synth.make_case("cont", dims, [130, 64], seed=2)
    assert (cont.block_table == np.arange(cont.block_table.size).reshape(cont.block_table.shape)).all()
    perm = synth.make_case("perm", dims, [130, 64], seed=2, layout="permuted", extra_pages=4)
    used = np.concatenate([perm.block_table[0, :3], perm.block_table[1, :1]])
    assert len(set(used.tolist())) == 4 and perm.num_pages == 8
    # the cache holds the first L - 1 tokens; every other slot is NaN with an out-of-range id
    rows = perm.c_pool.reshape(-1, dims.d_c)
    filled = ~np.isnan(f(rows)).all(axis=1)
    assert filled.sum() == 129 + 63
    assert (perm.id_pool.reshape(-1)[~filled] < 0).all()


def test_prefill_inputs_follow_the_recipe():
    """Packed prompts: offsets from the lengths, each prompt's pages distinct
    across the pool, the pool empty (NaN latents, ids -7), value ranges as in
    the decode workloads."""
    lens = [300, 0, 1, 129, 64]
    pc = synth.make_prefill_case("recipe", synth.dims_bf16(), lens, seed=3, extra_pages=2)
    assert list(pc.cu_seqlens) == [0, 300, 300, 301, 430, 494]
    assert pc.q.shape == (494, 16, 192) and pc.c.shape == (494, 256) and pc.kr.shape == (494, 64)
    P = pc.dims.page_size
    used = [int(p) for b, L in enumerate(lens) for p in pc.block_table[b, :(L + P - 1) // P]]
    assert len(used) == len(set(used)) == sum((L + P - 1) // P for L in lens)
    assert pc.num_pages == len(used) + 2 and max(used) < pc.num_pages
    assert np.isnan(f(pc.c_pool)).all() and (pc.id_pool == -7).all()
    assert (pc.ids >= 0).all() and (pc.ids < pc.dims.vocab).all()
    big = synth.case_prefill(batch=2, prompt=2048)
    c = f(big.c)
    assert abs(c.std() - 0.5) < 0.01 and abs(f(big.q).std() - 1.0) < 0.01


def test_prefill_ragged_lengths_and_embedding_inputs():
    pc = synth.case_prefill_ragged()
    L = pc.seq_lens
    assert L.min() >= 128 and L.max() <= 4096 and pc.dims.d_c == 192
    case = synth.make_case("emb", synth.dims_bf16(vocab=2000), [64], seed=4)
    emb, w_ue = synth.make_embedding(case, 256, seed=5)
    assert emb.shape == (2000, 256) and w_ue.shape == (256, 256)
    assert abs(f(emb).std() - 1.0) < 0.01 and abs(f(w_ue).std() - 1.0 / 16) < 0.002

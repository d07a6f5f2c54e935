"""GPU parity of one decode step through a whole attention layer
(eg_mla_layer_decode: projections, kv_norm and RoPE, append, gated latent
attention, output projection) against the fp64 layer oracle, through the C ABI.

Bounds, each fixed in advance by the arithmetic that produces the checked value:
  - the attention output u inside the layer (read where the call leaves it,
    eg_mla_layer_attn_offset) is held to the hot path's bf16 bound against the
    oracle's u of the same step: max-abs <= 1e-2 (per element 1e-2 max(1, |u|)
    for sequences shorter than the workloads' shortest context, as in the
    decode tests) and rel-L2 <= 5e-3;
  - the output y = W^O u is compared with W^O applied in fp64 to the GPU's own
    u: what remains is the projection's fp32 accumulation over K = H d_v terms
    (at most K 2^-24 sum_i |w_i u_i|) and the bf16 rounding of y (at most
    2^-8 |y|);
  - y against the oracle's y: rel-L2 <= 5e-3 (the decode's bound carried
    through a linear map);
  - the appended cache row (c^KV after kv_norm, the rotated k^R) lies within
    two bf16 units in the last place of the oracle's stored value (the
    projections are summed in a different order on the GPU, which can move a
    rounding by one unit).
"""
import numpy as np
import pytest
import torch

from oracle import egmla_oracle as orc
from paper_2509_16686_gb300 import _lib, device, synth

pytestmark = pytest.mark.gpu

BF16_MAX_ABS = 1e-2
BF16_REL_L2 = 5e-3


def rel_l2(got, ref):
    return float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))


def check_u(got, ref, where, scaled_abs):
    """The hot path's bf16 bound on the attention output."""
    assert np.isfinite(got).all(), where
    diff = np.abs(got - ref)
    bound = BF16_MAX_ABS * np.maximum(1.0, np.abs(ref)) if scaled_abs else BF16_MAX_ABS
    rel = rel_l2(got, ref)
    assert (diff <= bound).all() and rel <= BF16_REL_L2, f"{where} u: max_abs={diff.max():.3e} rel_l2={rel:.3e}"


def check_y(dl, lc, got_y, ref_y, where, batches=None):
    """y against W^O applied in fp64 to the GPU's u (rounding bound), and against
    the oracle's y (rel-L2)."""
    assert np.isfinite(got_y).all(), where
    u = device.output_f64(dl.attn_output()).reshape(dl.dc.batch, -1)
    w_o = orc.widen(lc.w_o, "bf16")
    bs = list(range(dl.dc.batch)) if batches is None else list(batches)
    y_u = u[bs] @ w_o.T
    acc = np.abs(u[bs]) @ np.abs(w_o).T
    k = w_o.shape[1]
    bound = 2.0 ** -8 * np.abs(y_u) + k * 2.0 ** -24 * acc
    diff = np.abs(got_y[bs] - y_u)
    assert (diff <= bound).all(), f"{where} y vs W^O u: worst {float((diff / bound).max()):.2f} of the bound"
    rel = rel_l2(got_y[bs], ref_y[bs])
    assert rel <= BF16_REL_L2, f"{where} y vs oracle: rel_l2={rel:.3e}"


def run_layer(lc, splits=0):
    dl = device.upload_layer(lc, num_splits=splits)
    dl.step()
    torch.cuda.synchronize()
    assert dl.dc.read_status() == 0
    return dl, device.output_f64(dl.y)


def check_appended_rows(dl, lc):
    """The new token's cache row against the oracle's stored c^KV and k^R."""
    step = orc.layer_step(lc)
    c_pool = dl.dc.c_pool.float().cpu().numpy()
    kr_pool = dl.dc.kr_pool.float().cpu().numpy()
    case = lc.case
    for b, pos in enumerate(case.positions()):
        page, slot = orc.paged_position(case.block_table, b, int(pos), case.dims.page_size)
        for got, ref_bits in ((c_pool[page, slot], step.c_new[b]), (kr_pool[page, slot], step.kr_new[b])):
            ref = orc.widen(ref_bits, "bf16")
            assert (np.abs(got - ref) <= 2 * 2.0 ** -8 * np.abs(ref) + 1e-30).all(), (b, np.abs(got - ref).max())


@pytest.mark.parametrize("d_c,gate", [(256, True), (192, True), (512, False)])
def test_layer_step_matches_oracle(gpu_lib, d_c, gate):
    case = synth.make_case("layer-small", synth.dims_bf16(d_c=d_c, vocab=3000, gate=gate), [70, 1, 200, 64, 129],
                           seed=31, latent_scale=0.5, layout="permuted", affine_ln=True, extra_pages=3)
    lc = synth.make_layer_case(case, 256, seed=32)
    ref = orc.layer_decode(lc)
    u_ref = orc.decode_unabsorbed(orc.layer_step(lc))
    for splits in (0, 3):
        dl, got = run_layer(lc, splits)
        where = f"layer d_c={d_c} gate={gate} splits={splits}"
        check_u(device.output_f64(dl.attn_output()), u_ref, where, scaled_abs=True)
        check_y(dl, lc, got, ref, where)
    check_appended_rows(dl, lc)


def test_layer_step_long_positions(gpu_lib):
    # rotation angles of positions in the tens of thousands
    case = synth.make_case("layer-long", synth.dims_bf16(vocab=3000), [30001, 16385], seed=33, latent_scale=0.5,
                           layout="permuted")
    lc = synth.make_layer_case(case, 512, seed=34)
    dl, got = run_layer(lc)
    check_u(device.output_f64(dl.attn_output()), orc.decode_unabsorbed(orc.layer_step(lc)), "long positions",
            scaled_abs=False)
    check_y(dl, lc, got, orc.layer_decode(lc), "layer long positions")
    check_appended_rows(dl, lc)


def test_layer_step_24_layer_model_shape_sampled(gpu_lib):
    # one layer of the 24-layer workload's shape: hidden 2048, batch 64 x 8192
    lc = synth.make_layer_case(synth.case_layer(0), 2048, seed=35)
    dl, got = run_layer(lc)
    sample = [0, 21, 37, 50, 63]
    step = orc.layer_step(lc)
    u_ref = orc.decode_unabsorbed(step, batches=sample)
    check_u(device.output_f64(dl.attn_output())[sample], u_ref[sample], "layer 2048 sampled", scaled_abs=False)
    check_y(dl, lc, got, orc.layer_decode(lc, batches=sample), "layer 2048 sampled", batches=sample)


def test_layer_group_shares_one_cache(gpu_lib):
    """Two layers of one layer group (Appendix H): the first projects, rotates and
    appends the shared c^KV, k^R; the second (share_kv) projects only its query
    and attends over the same cache with its own up-projections, gate table and
    output projection."""
    import dataclasses
    case_a = synth.make_case("group", synth.dims_bf16(vocab=3000), [300, 65, 1], seed=41, latent_scale=0.5,
                             layout="permuted", affine_ln=True)
    other = synth.make_case("group-b", synth.dims_bf16(vocab=3000), [300, 65, 1], seed=42, latent_scale=0.5,
                            layout="permuted", affine_ln=True)
    case_b = dataclasses.replace(case_a, gate_table=other.gate_table, ln_gamma=other.ln_gamma,
                                 ln_beta=other.ln_beta, w_uk=other.w_uk, w_uv=other.w_uv)
    lc_a = synth.make_layer_case(case_a, 256, seed=43)
    lc_b = synth.make_layer_case(case_b, 256, seed=44)
    dl_a = device.upload_layer(lc_a)
    dl_b = device.upload_layer(lc_b)
    for name in ("c_pool", "kr_pool", "id_pool", "block_table", "seq_lens", "positions", "ids_new"):
        setattr(dl_b.dc, name, getattr(dl_a.dc, name))
    dl_b.layer_dims = _lib.make_layer_dims(256, share_kv=True)
    dl_a.step()
    dl_b.step()
    torch.cuda.synchronize()
    assert dl_a.dc.read_status() == 0 and dl_b.dc.read_status() == 0
    check_u(device.output_f64(dl_a.attn_output()), orc.decode_unabsorbed(orc.layer_step(lc_a)), "group first layer",
            scaled_abs=True)
    check_y(dl_a, lc_a, device.output_f64(dl_a.y), orc.layer_decode(lc_a), "group first layer")
    # the second layer's u: its own step over the cache the first layer wrote
    check_u(device.output_f64(dl_b.attn_output()), orc.decode_unabsorbed(orc.layer_step(lc_b, kv_from=lc_a)),
            "group second layer", scaled_abs=True)
    check_y(dl_b, lc_b, device.output_f64(dl_b.y), orc.layer_decode(lc_b, kv_from=lc_a), "group second layer")
    # the cache holds the first layer's token once; a second append would have been the same row
    check_appended_rows(dl_a, lc_a)


def test_24_layer_chain_matches_chained_oracle(gpu_lib):
    """The 24-layer decoder step as the bench runs it (each layer's output y the
    next layer's input x), with 24 independently seeded layers (cache, gate
    table, weights), at a reduced batch and context.  Every layer is held to
    the layer bounds against the oracle applied to that layer's actual input
    (the GPU's y of the layer before, as stored in bf16); the chain's last
    output is compared with the oracle run through all 24 layers from the same
    first input, where each layer can add at most its own bound: rel-L2 <= 24 x
    5e-3 (reported, with the measured value, in the assertion message)."""
    import dataclasses
    n_layers, batch, ctx = 24, 4, 300
    lcs = []
    for k in range(n_layers):
        case = synth.case_layer(k, batch=batch, ctx=ctx, layout="permuted", extra_pages=2)
        lcs.append(synth.make_layer_case(case, 2048, seed=5000 + k))
    dls = [device.upload_layer(lc) for lc in lcs]
    for k in range(1, n_layers):
        dls[k].x = dls[k - 1].y
    for dl in dls:
        dl.step()
    torch.cuda.synchronize()
    for k, dl in enumerate(dls):
        assert dl.dc.read_status() == 0, k
    x_oracle = lcs[0].x
    for k, (lc, dl) in enumerate(zip(lcs, dls)):
        # layer k on its actual input
        x_gpu = device.bf16_tensor_to_bits(dl.x)
        lc_k = dataclasses.replace(lc, x=x_gpu)
        got = device.output_f64(dl.y)
        check_u(device.output_f64(dl.attn_output()), orc.decode_unabsorbed(orc.layer_step(lc_k)), f"chain layer {k}",
                scaled_abs=False)
        check_y(dl, lc_k, got, orc.layer_decode(lc_k), f"chain layer {k}")
        # the oracle's own chain, each y stored in the model dtype as the layer stores it
        y_oracle = orc.layer_decode(dataclasses.replace(lc, x=x_oracle))
        x_oracle = orc.store(y_oracle, "bf16")
    rel = rel_l2(got, y_oracle)
    assert rel <= n_layers * BF16_REL_L2, f"24-layer chain: rel_l2={rel:.3e}"


@pytest.mark.parametrize("n_out,k,batch,out_f32", [(3392, 2048, 64, True), (2048, 2048, 64, False),
                                                   (300, 136, 5, True), (128, 64, 16, False),
                                                   (1000, 520, 300, True), (3072, 2048, 1, True)])
def test_projection_gemm_matches_fp64(gpu_lib, n_out, k, batch, out_f32):
    """The layer's projection GEMM (eg_mla_debug_linear) against the product
    in fp64 of the same bf16 operands: the fp32 accumulation over k terms can
    move the sum by at most k 2^-24 sum_j |w_nj x_bj| (plus 2^-8 |out| for a
    bf16 result).  Shapes cover the layer's two projections, ragged tiles
    (n_out and k off the 128 and 64 multiples), a batch padded to 16, a batch
    beyond one launch's 256 rows, and one row; columns past n_out stay
    untouched."""
    rng = np.random.default_rng(n_out * 7 + k + batch)
    w = torch.from_numpy(rng.standard_normal((n_out, k)).astype(np.float32) * 0.05).to(torch.bfloat16).cuda()
    x = torch.from_numpy(rng.standard_normal((batch, k)).astype(np.float32)).to(torch.bfloat16).cuda()
    ldo = n_out + 8
    out = torch.full((batch, ldo), 7.0, dtype=torch.float32 if out_f32 else torch.bfloat16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    _lib.eg_mla_debug_linear(w, x, out, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    wf = w.double().cpu().numpy()
    xf = x.double().cpu().numpy()
    ref = xf @ wf.T
    got = out.double().cpu().numpy()
    bound = k * 2.0 ** -24 * (np.abs(xf) @ np.abs(wf).T)
    if not out_f32:
        bound = bound + 2.0 ** -8 * np.abs(ref)
    diff = np.abs(got[:, :n_out] - ref)
    assert (diff <= bound + 1e-30).all(), f"worst {float((diff / (bound + 1e-30)).max()):.2f} of the bound"
    assert (got[:, n_out:] == 7.0).all()

"""GPU parity of one decode step through a whole attention layer
(eg_mla_layer_decode: projections, kv_norm and RoPE, append, gated latent
attention, output projection) against the fp64 layer oracle, through the C ABI.

Bounds, derived from the arithmetic.  The attention output u inside the layer
carries the decode's bf16 error (rel-L2 <= 5e-3, the hot path's bound), and the
output y = W^O u sums the 2048 errors of u through a random weight row of unit
norm: each element's error is close to normal with standard deviation
rel-L2(u) * rms(y), and y itself is rounded to bf16.  So the layer output is
held to rel-L2 <= 5e-3 and, per element, |dy| <= 5 * 5e-3 * rms(y_ref) +
2^-8 |y_ref| (five standard deviations over ~10^4 outputs, plus one bf16
rounding).  The appended cache row (c^KV after kv_norm, the rotated k^R) is
within two bf16 units in the last place of the oracle's stored value (the
projections are summed in a different order on the GPU, which can move a
rounding by one unit).
"""
import numpy as np
import pytest
import torch

from oracle import egmla_oracle as orc
from paper_2509_16686_gb300 import _lib, device, synth

pytestmark = pytest.mark.gpu

BF16_REL_L2 = 5e-3


def check_bf16(got, ref, where):
    assert np.isfinite(got).all(), where
    diff = np.abs(got - ref)
    rel = float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))
    bound = 5 * BF16_REL_L2 * float(np.sqrt(np.mean(ref * ref))) + 2.0 ** -8 * np.abs(ref)
    worst = float((diff / bound).max())
    assert worst <= 1.0 and rel <= BF16_REL_L2, f"{where}: max_abs={diff.max():.3e} (x{worst:.2f} of bound) rel_l2={rel:.3e}"


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
    for splits in (0, 3):
        dl, got = run_layer(lc, splits)
        check_bf16(got, ref, f"layer d_c={d_c} gate={gate} splits={splits}")
    check_appended_rows(dl, lc)


def test_layer_step_long_positions(gpu_lib):
    # rotation angles of positions in the tens of thousands
    case = synth.make_case("layer-long", synth.dims_bf16(vocab=3000), [30001, 16385], seed=33, latent_scale=0.5,
                           layout="permuted")
    lc = synth.make_layer_case(case, 512, seed=34)
    dl, got = run_layer(lc)
    check_bf16(got, orc.layer_decode(lc), "layer long positions")
    check_appended_rows(dl, lc)


def test_layer_step_24_layer_model_shape_sampled(gpu_lib):
    # one layer of the 24-layer workload's shape: hidden 2048, batch 64 x 8192
    lc = synth.make_layer_case(synth.case_layer(0), 2048, seed=35)
    _, got = run_layer(lc)
    sample = [0, 37, 63]
    ref = orc.layer_decode(lc, batches=sample)
    check_bf16(got[sample], ref[sample], "layer 2048 sampled")


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
    check_bf16(device.output_f64(dl_a.y), orc.layer_decode(lc_a), "group first layer")
    check_bf16(device.output_f64(dl_b.y), orc.layer_decode(lc_b, kv_from=lc_a), "group second layer")
    # the cache holds the first layer's token once; a second append would have been the same row
    check_appended_rows(dl_a, lc_a)

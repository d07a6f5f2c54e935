"""GPU parity of eg_mla_gate_table (G = E W^UE^T for every vocabulary entry,
Section 3 Eqs. 3-4) against the oracle's gate_table_from_embedding, and of a
decode step gated through the table it computes (the EG-MLA form without a
precomputed table) against the oracle's decode.

Bound for the table: the GPU accumulates in fp32 and rounds each entry to bf16
once, so |got - ref| <= 2^-8 |ref| + 2^-16 max |ref| (half an ulp of bf16 plus
the fp32 sum).  The decode uses the hot path's bf16 bound."""
import numpy as np
import pytest
import torch

from oracle import egmla_oracle as orc
from paper_2509_16686_gb300 import _lib, device, synth

pytestmark = pytest.mark.gpu


def table_on_gpu(case, emb, w_ue):
    dims = device.dims_of(case)
    e = device.to_device_array(emb, "bf16", "cuda")
    w = device.to_device_array(w_ue, "bf16", "cuda")
    g = torch.full((case.dims.vocab, case.dims.d_c), float("nan"), dtype=torch.bfloat16, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    _lib.eg_mla_gate_table(dims, e, w, g, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return g


@pytest.mark.parametrize("d_c,d_e", [(256, 256), (192, 128), (256, 512), (512, 64)])
def test_gate_table_matches_oracle(gpu_lib, d_c, d_e):
    case = synth.make_case("gt", synth.dims_bf16(d_c=d_c, vocab=1000 + d_e), [70], seed=71, latent_scale=0.5)
    emb, w_ue = synth.make_embedding(case, d_e, seed=72)
    got = device.output_f64(table_on_gpu(case, emb, w_ue))
    ref = orc.gate_table_from_embedding(orc.widen(emb, "bf16"), orc.widen(w_ue, "bf16"))
    assert np.isfinite(got).all()
    bound = 2.0 ** -8 * np.abs(ref) + 2.0 ** -16 * np.abs(ref).max()
    assert (np.abs(got - ref) <= bound).all(), float((np.abs(got - ref) - bound).max())


@pytest.mark.parametrize("d_c", [256, 192])
def test_decode_gated_through_the_computed_table(gpu_lib, d_c):
    case = synth.make_case("gt-decode", synth.dims_bf16(d_c=d_c, vocab=2000), [300, 64, 1, 129], seed=73,
                           latent_scale=0.5, layout="permuted", affine_ln=True)
    emb, w_ue = synth.make_embedding(case, d_c, seed=74)
    dc = device.upload(case)
    dc.gate_table = table_on_gpu(case, emb, w_ue)
    got = device.output_f64(dc.step())
    torch.cuda.synchronize()
    assert dc.read_status() == 0
    ref_table = orc.gate_table_from_embedding(orc.widen(emb, "bf16"), orc.widen(w_ue, "bf16"))
    case.gate_table = orc.to_bf16_bits(ref_table)
    ref = orc.decode_unabsorbed(case)
    diff = np.abs(got - ref)
    rel = float(np.linalg.norm(got - ref) / np.linalg.norm(ref))
    assert (diff <= 1e-2 * np.maximum(1.0, np.abs(ref))).all() and rel <= 5e-3, (float(diff.max()), rel)

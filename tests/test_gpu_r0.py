"""GPU parity of the paper-literal (R0) gated decode, eg_mla_decode_r0,
against the fp64 oracle's `decode_r0` (gate and LayerNorm over the
H (d_n + d_v) = 4096 up-projected features of all heads, Section 3 Eq. 5
after Eq. 2, as the Appendix E listing does).

Bound: the hot path's bf16 bound, max-abs <= 1e-2 (per element
1e-2 max(1, |u|) for sequences shorter than the workloads' shortest context)
and rel-L2 <= 5e-3.  The GPU rounds the gated features z to bf16 once (as the
latent-gated kernel rounds its z), takes the LayerNorm statistics of the
rounded values in fp32 and rounds the output to bf16."""
import numpy as np
import pytest
import torch

from oracle import egmla_oracle as orc
from paper_2509_16686_gb300 import _lib, device, synth

pytestmark = pytest.mark.gpu


def rel_l2(got, ref):
    return float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))


def run_r0(case, r0):
    dc = device.upload(case)
    dc.append()
    w_ukv = device.to_device_array(r0.w_ukv, "bf16", "cuda")
    gate = device.to_device_array(r0.gate_r0, "bf16", "cuda")
    gamma = torch.from_numpy(r0.gamma).cuda()
    beta = torch.from_numpy(r0.beta).cuda()
    ws = torch.empty(_lib.eg_mla_decode_r0_workspace_size(dc.dims, case.batch, dc.block_table.shape[1],
                                                          case.num_pages), dtype=torch.uint8, device="cuda")
    out = torch.full((case.batch, 16, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    _lib.eg_mla_decode_r0(dc.dims, dc.q, dc.c_pool, dc.kr_pool, dc.id_pool, dc.block_table, dc.seq_lens, w_ukv,
                          gate, gamma, beta, out, ws, dc.status)
    torch.cuda.synchronize()
    return dc, device.output_f64(out)


@pytest.mark.parametrize("d_c,lens,affine", [(256, (70, 1, 200, 0, 129, 64), True), (192, (300, 65, 2), True),
                                             (256, (513,), False)])
def test_r0_decode_matches_oracle(gpu_lib, d_c, lens, affine):
    case = synth.make_case("r0", synth.dims_bf16(d_c=d_c, vocab=3000), list(lens), seed=51, latent_scale=0.5,
                           layout="permuted", affine_ln=True, extra_pages=3)
    r0 = synth.make_r0_inputs(case, seed=52, affine=affine)
    dc, got = run_r0(case, r0)
    assert dc.read_status() == 0
    ref = orc.decode_r0(case, gate_r0=orc.widen(r0.gate_r0, "bf16"), ln_gamma_r0=r0.gamma, ln_beta_r0=r0.beta)
    assert np.isfinite(got).all()
    diff = np.abs(got - ref)
    rel = rel_l2(got, ref)
    assert (diff <= 1e-2 * np.maximum(1.0, np.abs(ref))).all() and rel <= 5e-3, (diff.max(), rel)


def test_r0_out_of_range_id_is_reported(gpu_lib):
    case = synth.make_case("r0-oor", synth.dims_bf16(d_c=256, vocab=3000), [70, 20], seed=53, latent_scale=0.5,
                           layout="permuted")
    page = int(case.block_table[0, 0])
    case.id_pool[page, 5] = 3000   # one cached token with an id past the vocabulary
    r0 = synth.make_r0_inputs(case, seed=54)
    dc, got = run_r0(case, r0)
    assert dc.read_status() == _lib.EG_MLA_ERR_OUT_OF_RANGE
    assert np.isfinite(got).all()


def test_r0_batch_past_one_warp_of_sequences(gpu_lib):
    """40 sequences: the projection finds its pages with a prefix sum over the
    lanes 32 sequences at a time, so the second round of that scan is used."""
    rng = np.random.default_rng(55)
    lens = [int(x) for x in rng.integers(1, 300, size=40)]
    lens[7], lens[33] = 0, 64
    case = synth.make_case("r0-b40", synth.dims_bf16(d_c=192, vocab=3000), lens, seed=56, latent_scale=0.5,
                           layout="permuted", affine_ln=True, extra_pages=5)
    r0 = synth.make_r0_inputs(case, seed=57)
    dc, got = run_r0(case, r0)
    assert dc.read_status() == 0
    ref = orc.decode_r0(case, gate_r0=orc.widen(r0.gate_r0, "bf16"), ln_gamma_r0=r0.gamma, ln_beta_r0=r0.beta)
    diff = np.abs(got - ref)
    assert (diff <= 1e-2 * np.maximum(1.0, np.abs(ref))).all() and rel_l2(got, ref) <= 5e-3, (diff.max(),)


def test_r0_pages_shared_between_sequences(gpu_lib):
    """A page in two sequences' block tables (a shared prefix) is projected for
    each of them; both write the same gated values, and each sequence's logits
    are its own."""
    case = synth.make_case("r0-shared", synth.dims_bf16(d_c=256, vocab=3000), [300, 200, 150], seed=58,
                           latent_scale=0.5, layout="permuted", affine_ln=True)
    case.block_table[1, 0] = case.block_table[0, 0]
    case.block_table[2, 1] = case.block_table[0, 2]
    r0 = synth.make_r0_inputs(case, seed=59)
    dc, got = run_r0(case, r0)
    assert dc.read_status() == 0
    ref = orc.decode_r0(case, gate_r0=orc.widen(r0.gate_r0, "bf16"), ln_gamma_r0=r0.gamma, ln_beta_r0=r0.beta)
    diff = np.abs(got - ref)
    assert (diff <= 1e-2 * np.maximum(1.0, np.abs(ref))).all() and rel_l2(got, ref) <= 5e-3, (diff.max(),)


def test_r0_full_size_sampled(gpu_lib):
    """The R0 bench workload itself (8 sequences x 4096 tokens, d_c 256,
    vocabulary 32000, the bench's seeds and launch): sequences 0 and 5, every
    head, against the oracle."""
    case = synth.case_c4k(batch=8, ctx=4096, keep_logical=False)
    r0 = synth.make_r0_inputs(case, seed=61)
    dc, got = run_r0(case, r0)
    assert dc.read_status() == 0
    picked = [0, 5]
    ref = orc.decode_r0(case, gate_r0=orc.widen(r0.gate_r0, "bf16"), ln_gamma_r0=r0.gamma, ln_beta_r0=r0.beta,
                        batches=picked)
    g, r = got[picked], ref[picked]
    diff = np.abs(g - r)
    assert (diff <= 1e-2 * np.maximum(1.0, np.abs(r))).all() and rel_l2(g, r) <= 5e-3, (diff.max(), rel_l2(g, r))

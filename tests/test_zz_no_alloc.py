"""eg_mla_decode_static: the decode entry that runs on the library's static
scratch array instead of a caller workspace.

The GPU tests call it through the C ABI twice in a row on the same inputs and
compare both results with eg_mla_decode (caller workspace) on the same cache,
within the parity tolerances of the hot path.  The file is collected last so
that the static-scratch calls also run after every other test in one process.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2509_16686_gb300 import _lib, device, synth

BF16_MAX_ABS = 1e-2
BF16_REL_L2 = 5e-3
F32_REL_L2 = 1e-5


def rel_l2(got, ref):
    return float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))


def static_decode(dc, out):
    _lib.eg_mla_decode_static(dc.dims, dc.q, dc.c_pool, dc.kr_pool, dc.id_pool, dc.block_table, dc.seq_lens,
                              dc.max_seq_len, dc.gate_table, dc.ln_gamma, dc.ln_beta, dc.w_uk, dc.w_uv, out,
                              dc.num_splits, dc.status)


def compare_two_static_calls(case, num_splits, check):
    dc = device.upload(case, num_splits=num_splits)
    dc.step()  # append the new token, then decode with the caller workspace
    torch.cuda.synchronize()
    assert dc.read_status() == 0
    ref = device.output_f64(dc.out)
    outs = []
    for _ in range(2):
        out = torch.full_like(dc.out, float("nan"))
        static_decode(dc, out)
        torch.cuda.synchronize()
        assert dc.read_status() == 0
        outs.append(device.output_f64(out))
    for got in outs:
        assert np.isfinite(got).all()
        check(got, ref)
    return outs


def check_bf16(got, ref):
    assert np.abs(got - ref).max() <= BF16_MAX_ABS and rel_l2(got, ref) <= BF16_REL_L2


def check_f32(got, ref):
    assert rel_l2(got, ref) <= F32_REL_L2


@pytest.mark.gpu
def test_static_scratch_decode_matches_workspace_decode_bf16(gpu_lib):
    dims = synth.dims_bf16(d_c=256, vocab=3000, gate=True)
    case = synth.make_case("static-bf16", dims, [1000, 37, 0, 513, 64], seed=23, latent_scale=0.5,
                           layout="permuted", affine_ln=True, extra_pages=5)
    compare_two_static_calls(case, 7, check_bf16)


@pytest.mark.gpu
def test_static_scratch_decode_matches_workspace_decode_default_splits(gpu_lib):
    dims = synth.dims_bf16(d_c=192, vocab=3000, gate=True)
    case = synth.make_case("static-bf16-192", dims, [300, 2049, 129], seed=24, latent_scale=0.5,
                           layout="permuted", affine_ln=True, extra_pages=3)
    compare_two_static_calls(case, 0, check_bf16)


@pytest.mark.gpu
def test_static_scratch_decode_matches_workspace_decode_fp32(gpu_lib):
    compare_two_static_calls(synth.case_tiny(), 3, check_f32)


def test_static_scratch_limit_is_rejected_before_launch():
    """A problem whose workspace exceeds the static array is refused on the host
    (no device pointer is touched, so this runs without a GPU)."""
    lib = _lib.load()
    dims = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    splits = 2000
    need = lib.eg_mla_decode_workspace_size(ctypes.byref(dims), 8, splits)
    assert need > _lib.STATIC_SCRATCH_BYTES
    null = None
    rc = lib.eg_mla_decode_static(ctypes.byref(dims), null, null, null, null, null, 1, null, 64, 8, 1, null,
                                  null, null, null, null, null, splits, null, null)
    assert rc == _lib.EG_MLA_ERR_SCRATCH_LIMIT
    assert b"static scratch" in lib.eg_mla_status_string(rc)
    # a negative split count is an argument error, as for eg_mla_decode
    rc = lib.eg_mla_decode_static(ctypes.byref(dims), null, null, null, null, null, 1, null, 64, 8, 1, null,
                                  null, null, null, null, null, -1, null, null)
    assert rc == _lib.EG_MLA_ERR_INVALID_ARG

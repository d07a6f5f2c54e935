"""Host-side checks of the C ABI that need no GPU: the library builds and loads,
exports every symbol include/egmla.h declares, and its host-only calls and
argument validation behave as documented."""
import ctypes
import os
import re

import pytest

from paper_2509_16686_gb300 import _lib

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    src = open(os.path.join(ROOT, "include", "egmla.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(eg_mla_[a-z_0-9]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    return _lib.load()


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 7
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(_lib.EXPORTED) == names


def test_dims_struct_matches_header():
    src = open(os.path.join(ROOT, "include", "egmla.h")).read()
    body = re.search(r"typedef struct \{(.*?)\} eg_mla_dims;", src, flags=re.S).group(1)
    fields = re.findall(r"(int32_t|float)\s+([a-z_0-9, ]+);", body)
    flat = []
    for ty, names in fields:
        for n in names.split(","):
            flat.append((ty, n.strip()))
    assert [n for _, n in flat] == [n for n, _ in _lib.EgMlaDims._fields_]
    assert ctypes.sizeof(_lib.EgMlaDims) == 4 * len(flat)


def test_status_strings(lib):
    for code in range(0, -7, -1):
        assert lib.eg_mla_status_string(code)
    assert b"unknown" in lib.eg_mla_status_string(42)


def test_kv_bytes_per_token():
    d = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    assert _lib.eg_mla_kv_bytes_per_token(d, 1) == 644
    assert _lib.eg_mla_kv_bytes_per_token(d, 24) == 24 * 644
    d = _lib.make_dims(16, 128, 64, 128, 512, 50000, gate=False)
    assert _lib.eg_mla_kv_bytes_per_token(d, 1) == 1152
    d = _lib.make_dims(4, 32, 16, 32, 64, 1000, dtype="fp32")
    assert _lib.eg_mla_kv_bytes_per_token(d, 1) == (64 + 16) * 4 + 4


def test_workspace_size_and_shape_support():
    d = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    n1 = _lib.eg_mla_decode_workspace_size(d, 8, 152)
    n2 = _lib.eg_mla_decode_workspace_size(d, 8, 304)
    assert n2 > n1 > 0 and n1 % 256 == 0
    # partials: (splits + batch) x heads x (d_c + 2) floats dominate
    assert n1 >= (152 + 8) * 16 * (256 + 2) * 4
    bad = _lib.make_dims(8, 128, 64, 128, 256, 32000)          # bf16 path is built for 16 heads
    assert _lib.load().eg_mla_decode_workspace_size(ctypes.byref(bad), 8, 152) == 0
    bad = _lib.make_dims(16, 128, 64, 128, 512, 32000, gate=True)  # gated d_c 512 not built
    assert _lib.load().eg_mla_decode_workspace_size(ctypes.byref(bad), 8, 152) == 0


def test_invalid_arguments_are_rejected_before_launch(lib):
    d = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    P = ctypes.c_void_p
    fake = P(0x10000)  # never dereferenced: validation fails first
    rc = lib.eg_mla_decode(ctypes.byref(d), fake, None, fake, fake, fake, 4, fake, 256, 2, 8, fake, None, None,
                           fake, fake, fake, 152, fake, 1 << 20, None, None)
    assert rc == _lib.EG_MLA_ERR_INVALID_ARG
    # max_seq_len beyond the block table's reach
    rc = lib.eg_mla_decode(ctypes.byref(d), fake, fake, fake, fake, fake, 4, fake, 257, 2, 8, fake, None, None,
                           fake, fake, fake, 152, fake, 1 << 20, None, None)
    assert rc == _lib.EG_MLA_ERR_INVALID_ARG
    # workspace too small
    rc = lib.eg_mla_decode(ctypes.byref(d), fake, fake, fake, fake, fake, 4, fake, 256, 2, 8, fake, None, None,
                           fake, fake, fake, 152, fake, 16, None, None)
    assert rc == _lib.EG_MLA_ERR_WORKSPACE
    # misaligned cache pool
    rc = lib.eg_mla_decode(ctypes.byref(d), fake, P(0x10008), fake, fake, fake, 4, fake, 256, 2, 8, fake, None,
                           None, fake, fake, fake, 152, fake, 1 << 20, None, None)
    assert rc == _lib.EG_MLA_ERR_INVALID_ARG
    # unsupported shape
    d2 = _lib.make_dims(16, 128, 32, 128, 256, 32000)
    rc = lib.eg_mla_decode(ctypes.byref(d2), fake, fake, fake, fake, fake, 4, fake, 256, 2, 8, fake, None, None,
                           fake, fake, fake, 152, fake, 1 << 20, None, None)
    assert rc == _lib.EG_MLA_ERR_UNSUPPORTED
    # append: null pool
    rc = lib.eg_mla_append_latent(ctypes.byref(d), None, fake, fake, fake, fake, fake, fake, 4, fake, 2, 8, None,
                                  None)
    assert rc == _lib.EG_MLA_ERR_INVALID_ARG


def test_library_has_no_oracle_dependency():
    # the product path must not reach the test oracle
    pkg = os.path.join(ROOT, "paper_2509_16686_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in text and "from oracle" not in text, f


def test_layer_workspace_size():
    d = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    ld = _lib.make_layer_dims(2048)
    n = _lib.eg_mla_layer_workspace_size(d, ld, 64, 152)
    dec = _lib.eg_mla_decode_workspace_size(d, 64, 152)
    # the decode workspace, the fp32 projections and bf16 q, c, k^R, u
    assert n >= dec + 64 * (16 * 192 + 320) * 4 + 64 * (16 * 192 + 256 + 64 + 16 * 128) * 2
    assert n % 256 == 0
    f32 = _lib.make_dims(4, 32, 16, 32, 64, 1000, dtype="fp32")
    assert _lib.load().eg_mla_layer_workspace_size(ctypes.byref(f32), ctypes.byref(ld), 4, 8) == 0
    assert _lib.load().eg_mla_layer_workspace_size(ctypes.byref(d), None, 4, 8) == 0


def test_layer_decode_rejects_before_launch(lib):
    d = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    ld = _lib.make_layer_dims(2048)
    fake = 0x10000  # 256-byte aligned, never dereferenced: validation fails first
    w = _lib.EgMlaLayerWeights(*([fake] * 8))
    P = ctypes.c_void_p

    def call(dims=d, layer=ld, weights=w, x=fake, batch=4, ws_bytes=1 << 20):
        return lib.eg_mla_layer_decode(ctypes.byref(dims), ctypes.byref(layer), ctypes.byref(weights), P(x),
                                       P(fake), P(fake), P(fake), P(fake), P(fake), P(fake), 4, P(fake), 256, batch,
                                       8, P(fake), 152, P(fake), ws_bytes, None, None)
    assert call(dims=_lib.make_dims(4, 32, 16, 32, 64, 1000, dtype="fp32")) == _lib.EG_MLA_ERR_UNSUPPORTED
    assert call(layer=_lib.make_layer_dims(2044)) == _lib.EG_MLA_ERR_UNSUPPORTED
    assert call(x=0) == _lib.EG_MLA_ERR_INVALID_ARG
    assert call(x=fake + 8) == _lib.EG_MLA_ERR_INVALID_ARG              # 16-byte alignment
    assert call(ws_bytes=1 << 20) == _lib.EG_MLA_ERR_WORKSPACE         # far below the layer's workspace
    assert call(batch=0) == _lib.EG_MLA_OK                              # nothing to do, nothing launched


def test_fault_entry_validates_its_arguments(lib):
    # host-only: no launch happens here; cta < 0 restores normal operation
    assert lib.eg_mla_debug_set_fault(0, -1, 1_000_000) == _lib.EG_MLA_ERR_INVALID_ARG
    assert lib.eg_mla_debug_set_fault(0, 1, 10) == _lib.EG_MLA_ERR_INVALID_ARG
    assert lib.eg_mla_debug_set_fault(0, 1, 3_000_000_000) == _lib.EG_MLA_ERR_INVALID_ARG
    assert lib.eg_mla_debug_set_fault(0, 1, 1_000_000) == _lib.EG_MLA_OK
    assert lib.eg_mla_debug_set_fault(-1, 0, 0) == _lib.EG_MLA_OK


def test_layer_attention_offset_is_inside_the_workspace(lib):
    dims = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    layer = _lib.make_layer_dims(2048)
    ws = _lib.eg_mla_layer_workspace_size(dims, layer, 64, 152)
    off = _lib.eg_mla_layer_attn_offset(dims, layer, 64, 152)
    assert 0 < off and off % 256 == 0 and off + 64 * 16 * 128 * 2 <= ws


# --------------------------------------------------------------------------- prefill: host-side checks
def _prefill_call(lib, dims, **kw):
    """eg_mla_prefill with fake, aligned device addresses; each case makes one
    host check fail, so the call returns before anything is launched."""
    P = lambda v: ctypes.c_void_p(v)
    a = dict(q=0x1000, c=0x2000, kr=0x3000, ids=0x4000, cu=0x5000, batch=2, total=100, max_len=60, gate=0x6000,
             gamma=None, beta=None, w_uk=0x7000, w_uv=0x8000, out=0x9000, c_pool=None, kr_pool=None, id_pool=None,
             bt=None, max_pages=0, num_pages=0, ws=0xA000, ws_bytes=1 << 30, status=None)
    a.update(kw)
    return lib.eg_mla_prefill(ctypes.byref(dims), P(a["q"]), P(a["c"]), P(a["kr"]), P(a["ids"]), P(a["cu"]),
                              a["batch"], a["total"], a["max_len"], P(a["gate"]), P(a["gamma"]), P(a["beta"]),
                              P(a["w_uk"]), P(a["w_uv"]), P(a["out"]), P(a["c_pool"]), P(a["kr_pool"]),
                              P(a["id_pool"]), P(a["bt"]), a["max_pages"], a["num_pages"], P(a["ws"]),
                              ctypes.c_size_t(a["ws_bytes"]), P(a["status"]), None)


def test_prefill_workspace_size(lib):
    d = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    n = _lib.eg_mla_prefill_workspace_size(d, 8, 32768)
    # launch order (8 int32), c~ (32768 x 256 bf16), keys and values (32768 x 16 x 256 bf16)
    assert n == 256 + 32768 * 256 * 2 + 32768 * 16 * 256 * 2
    assert lib.eg_mla_prefill_workspace_size(ctypes.byref(_lib.make_dims(16, 64, 64, 128, 256, 32000)), 8, 100) == 0


def test_prefill_rejects_bad_arguments(lib):
    d = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    assert _prefill_call(lib, d, batch=0) == _lib.EG_MLA_OK                 # nothing to do
    assert _prefill_call(lib, d, total=0) == _lib.EG_MLA_OK
    assert _prefill_call(lib, d, batch=-1) == _lib.EG_MLA_ERR_INVALID_ARG
    assert _prefill_call(lib, d, max_len=0) == _lib.EG_MLA_ERR_INVALID_ARG
    assert _prefill_call(lib, d, max_len=101) == _lib.EG_MLA_ERR_INVALID_ARG  # longer than all tokens
    assert _prefill_call(lib, d, q=0) == _lib.EG_MLA_ERR_INVALID_ARG
    assert _prefill_call(lib, d, ids=0) == _lib.EG_MLA_ERR_INVALID_ARG       # gated: ids needed
    assert _prefill_call(lib, d, gate=0) == _lib.EG_MLA_ERR_INVALID_ARG
    assert _prefill_call(lib, d, out=0x9008) == _lib.EG_MLA_ERR_INVALID_ARG  # 16-byte alignment
    assert _prefill_call(lib, d, c_pool=0xB000) == _lib.EG_MLA_ERR_INVALID_ARG  # pool without block table
    assert _prefill_call(lib, d, ws_bytes=1000) == _lib.EG_MLA_ERR_WORKSPACE
    assert _prefill_call(lib, d, ws=0xA010) == _lib.EG_MLA_ERR_WORKSPACE     # 256-byte alignment
    for bad in (_lib.make_dims(16, 64, 64, 128, 256, 32000),                   # d_nope 64
                _lib.make_dims(16, 128, 32, 128, 256, 32000),                  # d_rope 32
                _lib.make_dims(16, 128, 64, 128, 200, 32000),                  # d_c not a multiple of 64
                _lib.make_dims(16, 128, 64, 128, 576, 32000),                  # d_c above 512
                _lib.make_dims(4, 128, 64, 128, 256, 1000, dtype="fp32")):     # fp32
        assert _prefill_call(lib, bad) == _lib.EG_MLA_ERR_UNSUPPORTED
    # gate off: ids and gate table may be null
    d_off = _lib.make_dims(16, 128, 64, 128, 256, 32000, gate=False)
    assert _prefill_call(lib, d_off, ids=0, gate=0, ws_bytes=1000) == _lib.EG_MLA_ERR_WORKSPACE


# --------------------------------------------------------------------------- R0 decode: host-side checks
def _r0_call(lib, dims, **kw):
    """eg_mla_decode_r0 with fake, aligned device addresses; each case makes one
    host check fail, so the call returns before anything is launched."""
    P = lambda v: ctypes.c_void_p(v)
    a = dict(q=0x1000, c_pool=0x2000, kr_pool=0x3000, id_pool=0x4000, bt=0x5000, max_pages=4, seq_lens=0x6000,
             batch=2, num_pages=8, w_ukv=0x7000, gate=0x8000, gamma=None, beta=None, out=0x9000, ws=0xA000,
             ws_bytes=1 << 30, status=None)
    a.update(kw)
    return lib.eg_mla_decode_r0(ctypes.byref(dims), P(a["q"]), P(a["c_pool"]), P(a["kr_pool"]), P(a["id_pool"]),
                                P(a["bt"]), a["max_pages"], P(a["seq_lens"]), a["batch"], a["num_pages"],
                                P(a["w_ukv"]), P(a["gate"]), P(a["gamma"]), P(a["beta"]), P(a["out"]), P(a["ws"]),
                                ctypes.c_size_t(a["ws_bytes"]), P(a["status"]), None)


def test_r0_workspace_size(lib):
    d = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    # gated values (16 x 128 bf16 per pool row), row statistics (2 fp32), and
    # 16 fp32 logits per (sequence, position) of the block table; 256-byte pieces
    rows, positions = 512 * 64, 8 * 64 * 64
    expect = rows * 16 * 128 * 2 + rows * 8 + positions * 16 * 4
    assert _lib.eg_mla_decode_r0_workspace_size(d, 8, 64, 512) == expect
    assert _lib.eg_mla_decode_r0_workspace_size(d, 8, 64, 512) < _lib.eg_mla_decode_r0_workspace_size(d, 9, 64, 512)
    for bad in (_lib.make_dims(16, 128, 64, 128, 512, 32000, gate=False),   # d_c 512
                _lib.make_dims(16, 64, 64, 64, 256, 32000),                 # d_nope, d_v 64
                _lib.make_dims(4, 32, 16, 32, 64, 1000, dtype="fp32")):     # fp32
        assert lib.eg_mla_decode_r0_workspace_size(ctypes.byref(bad), 8, 64, 512) == 0
    assert lib.eg_mla_decode_r0_workspace_size(ctypes.byref(d), 8, 0, 512) == 0       # no block table
    assert lib.eg_mla_decode_r0_workspace_size(ctypes.byref(d), 8, 64, 0) == 0        # no pool


def test_r0_rejects_bad_arguments(lib):
    d = _lib.make_dims(16, 128, 64, 128, 256, 32000)
    assert _r0_call(lib, d, batch=0) == _lib.EG_MLA_OK                       # nothing to do
    assert _r0_call(lib, d, batch=-1) == _lib.EG_MLA_ERR_INVALID_ARG
    assert _r0_call(lib, d, max_pages=0) == _lib.EG_MLA_ERR_INVALID_ARG
    assert _r0_call(lib, d, num_pages=0) == _lib.EG_MLA_ERR_INVALID_ARG
    for name in ("q", "c_pool", "kr_pool", "id_pool", "bt", "seq_lens", "w_ukv", "gate", "out"):
        assert _r0_call(lib, d, **{name: 0}) == _lib.EG_MLA_ERR_INVALID_ARG, name
    assert _r0_call(lib, d, out=0x9008) == _lib.EG_MLA_ERR_INVALID_ARG      # 16-byte alignment
    assert _r0_call(lib, d, gate=0x8004) == _lib.EG_MLA_ERR_INVALID_ARG
    need = _lib.eg_mla_decode_r0_workspace_size(d, 2, 4, 8)
    assert _r0_call(lib, d, ws_bytes=need - 1) == _lib.EG_MLA_ERR_WORKSPACE
    assert _r0_call(lib, d, ws=0xA010) == _lib.EG_MLA_ERR_WORKSPACE          # 256-byte alignment
    assert _r0_call(lib, d, ws=0) == _lib.EG_MLA_ERR_WORKSPACE
    for bad in (_lib.make_dims(16, 128, 64, 128, 512, 32000, gate=False),
                _lib.make_dims(16, 128, 64, 128, 128, 32000),                 # d_c 128
                _lib.make_dims(4, 32, 16, 32, 64, 1000, dtype="fp32")):
        assert _r0_call(lib, bad) == _lib.EG_MLA_ERR_UNSUPPORTED

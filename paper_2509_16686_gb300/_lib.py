"""ctypes binding of libegmla (include/egmla.h).

Argument marshalling only: torch tensors are passed as raw device pointers and
the current torch CUDA stream as the stream handle; every step of the decode
path runs in the library's kernels.  There is no fallback: if the library
cannot be built or loaded, ``load()`` raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional

import torch

from . import build as _build

EG_MLA_OK = 0
EG_MLA_ERR_INVALID_ARG = -1
EG_MLA_ERR_UNSUPPORTED = -2
EG_MLA_ERR_CUDA = -3
EG_MLA_ERR_OUT_OF_RANGE = -4
EG_MLA_ERR_TIMEOUT = -5
EG_MLA_ERR_WORKSPACE = -6
EG_MLA_ERR_SCRATCH_LIMIT = -7

# size of the library's static scratch array (EG_MLA_STATIC_SCRATCH_BYTES)
STATIC_SCRATCH_BYTES = 16 << 20

EG_MLA_BF16 = 0
EG_MLA_FP32 = 1
EG_MLA_GATE_NONE = 0
EG_MLA_GATE_MUL_LN = 1
EG_MLA_GATE_MUL = 2      # ablation: LayerNorm removed
EG_MLA_GATE_ADD_LN = 3   # ablation: (*) replaced by +
GATE_MODES = {"mul_ln": EG_MLA_GATE_MUL_LN, "mul": EG_MLA_GATE_MUL, "add_ln": EG_MLA_GATE_ADD_LN}

EXPORTED = [
    "eg_mla_append_latent",
    "eg_mla_default_num_splits",
    "eg_mla_decode_workspace_size",
    "eg_mla_decode",
    "eg_mla_decode_static",
    "eg_mla_step",
    "eg_mla_decode_r0_workspace_size",
    "eg_mla_decode_r0",
    "eg_mla_prefill_workspace_size",
    "eg_mla_prefill",
    "eg_mla_gate_table",
    "eg_mla_kv_bytes_per_token",
    "eg_mla_status_string",
    "eg_mla_debug_gather",
    "eg_mla_debug_linear",
    "eg_mla_debug_linear_plan",
    "eg_mla_profile_begin",
    "eg_mla_profile_end",
    "eg_mla_debug_set_trace",
    "eg_mla_debug_set_fault",
    "eg_mla_layer_workspace_size",
    "eg_mla_layer_attn_offset",
    "eg_mla_layer_decode",
]


class EgMlaDims(ctypes.Structure):
    _fields_ = [
        ("num_heads", ctypes.c_int32),
        ("d_nope", ctypes.c_int32),
        ("d_rope", ctypes.c_int32),
        ("d_v", ctypes.c_int32),
        ("d_c", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
        ("vocab", ctypes.c_int32),
        ("dtype", ctypes.c_int32),
        ("gate_mode", ctypes.c_int32),
        ("softmax_scale", ctypes.c_float),
        ("ln_eps", ctypes.c_float),
    ]


class EgMlaError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {status_string(code)} ({code})")


_lock = threading.Lock()
_handle: Optional[ctypes.CDLL] = None


def _declare(lib: ctypes.CDLL) -> None:
    P, I32, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    D = ctypes.POINTER(EgMlaDims)
    lib.eg_mla_append_latent.argtypes = [D, P, P, P, P, P, P, P, I32, P, I32, I32, P, P]
    lib.eg_mla_append_latent.restype = ctypes.c_int
    lib.eg_mla_default_num_splits.argtypes = [ctypes.POINTER(I32)]
    lib.eg_mla_default_num_splits.restype = ctypes.c_int
    lib.eg_mla_decode_workspace_size.argtypes = [D, I32, I32]
    lib.eg_mla_decode_workspace_size.restype = SZ
    lib.eg_mla_decode.argtypes = [D, P, P, P, P, P, I32, P, I32, I32, I32, P, P, P, P, P, P, I32, P, SZ, P, P]
    lib.eg_mla_decode.restype = ctypes.c_int
    lib.eg_mla_decode_static.argtypes = [D, P, P, P, P, P, I32, P, I32, I32, I32, P, P, P, P, P, P, I32, P, P]
    lib.eg_mla_decode_static.restype = ctypes.c_int
    lib.eg_mla_step.argtypes = [D, P, P, P, P, P, P, P, P, P, I32, P, I32, I32, I32, P, P, P, P, P, P, I32, P, SZ,
                                P, P]
    lib.eg_mla_step.restype = ctypes.c_int
    lib.eg_mla_decode_r0_workspace_size.argtypes = [D, I32, I32, I32]
    lib.eg_mla_decode_r0_workspace_size.restype = SZ
    lib.eg_mla_decode_r0.argtypes = [D, P, P, P, P, P, I32, P, I32, I32, P, P, P, P, P, P, SZ, P, P]
    lib.eg_mla_decode_r0.restype = ctypes.c_int
    lib.eg_mla_prefill_workspace_size.argtypes = [D, I32, I32]
    lib.eg_mla_prefill_workspace_size.restype = SZ
    lib.eg_mla_prefill.argtypes = [D, P, P, P, P, P, I32, I32, I32, P, P, P, P, P, P, P, P, P, P, I32, I32,
                                   P, SZ, P, P]
    lib.eg_mla_prefill.restype = ctypes.c_int
    lib.eg_mla_gate_table.argtypes = [D, I32, P, P, P, P, P]
    lib.eg_mla_gate_table.restype = ctypes.c_int
    lib.eg_mla_debug_linear.argtypes = [P, I32, I32, P, I32, P, I32, I32, P, P]
    lib.eg_mla_debug_linear.restype = ctypes.c_int
    lib.eg_mla_debug_linear_plan.argtypes = [I32, I32, I32, ctypes.POINTER(I32), ctypes.POINTER(I32),
                                             ctypes.POINTER(I32)]
    lib.eg_mla_debug_linear_plan.restype = ctypes.c_int
    lib.eg_mla_kv_bytes_per_token.argtypes = [D, I32, ctypes.POINTER(ctypes.c_int64)]
    lib.eg_mla_kv_bytes_per_token.restype = ctypes.c_int
    lib.eg_mla_status_string.argtypes = [ctypes.c_int]
    lib.eg_mla_status_string.restype = ctypes.c_char_p
    lib.eg_mla_debug_gather.argtypes = [D, P, P, P, P, I32, P, I32, I32, I32, P, P, P, P, P, I32, P, SZ, P, P]
    lib.eg_mla_debug_gather.restype = ctypes.c_int
    lib.eg_mla_profile_begin.argtypes = [I32]
    lib.eg_mla_profile_begin.restype = ctypes.c_int
    lib.eg_mla_profile_end.argtypes = [ctypes.POINTER(ctypes.c_double), ctypes.POINTER(I32)]
    lib.eg_mla_profile_end.restype = ctypes.c_int
    lib.eg_mla_debug_set_trace.argtypes = [P, ctypes.c_int64, I32]
    lib.eg_mla_debug_set_trace.restype = ctypes.c_int
    lib.eg_mla_debug_set_fault.argtypes = [I32, I32, ctypes.c_int64]
    lib.eg_mla_debug_set_fault.restype = ctypes.c_int
    LD, LW = ctypes.POINTER(EgMlaLayerDims), ctypes.POINTER(EgMlaLayerWeights)
    lib.eg_mla_layer_workspace_size.argtypes = [D, LD, I32, I32]
    lib.eg_mla_layer_workspace_size.restype = SZ
    lib.eg_mla_layer_attn_offset.argtypes = [D, LD, I32, I32]
    lib.eg_mla_layer_attn_offset.restype = SZ
    lib.eg_mla_layer_decode.argtypes = [D, LD, LW, P, P, P, P, P, P, P, I32, P, I32, I32, I32, P, I32, P, SZ, P, P]
    lib.eg_mla_layer_decode.restype = ctypes.c_int


def library_path() -> str:
    return _build.LIB


def load(build_if_needed: bool = True) -> ctypes.CDLL:
    """Load (building first if needed) the in-tree libegmla.so."""
    global _handle
    with _lock:
        if _handle is None:
            path = _build.build() if build_if_needed else _build.LIB
            if not os.path.exists(path):
                raise RuntimeError(f"libegmla not built: {path}")
            lib = ctypes.CDLL(path)
            _declare(lib)
            _handle = lib
    return _handle


def status_string(code: int) -> str:
    if _handle is None:
        return f"status {code}"
    return _handle.eg_mla_status_string(code).decode()


def _check(code: int, where: str) -> None:
    if code != EG_MLA_OK:
        raise EgMlaError(code, where)

class EgMlaLayerDims(ctypes.Structure):
    _fields_ = [
        ("n_embd", ctypes.c_int32),
        ("rope_theta", ctypes.c_float),
        ("rms_eps", ctypes.c_float),
        ("share_kv", ctypes.c_int32),
    ]


class EgMlaLayerWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("w_qkv_a", "kv_norm_w", "w_o", "gate_table", "ln_gamma", "ln_beta",
                                                "w_uk", "w_uv")]


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("device tensor expected")
    if not t.is_contiguous():
        raise ValueError("contiguous tensor expected")
    return t.data_ptr()


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def make_dims(num_heads, d_nope, d_rope, d_v, d_c, vocab, dtype="bf16", gate=True, page_size=64,
              softmax_scale=0.0, ln_eps=1e-5, gate_op="mul_ln") -> EgMlaDims:
    """gate False: plain MLA; gate True: gate operation `gate_op` ("mul_ln",
    or the ablations "mul" and "add_ln")."""
    return EgMlaDims(num_heads, d_nope, d_rope, d_v, d_c, page_size, vocab,
                     EG_MLA_BF16 if dtype == "bf16" else EG_MLA_FP32,
                     GATE_MODES[gate_op] if gate else EG_MLA_GATE_NONE, softmax_scale, ln_eps)


def eg_mla_default_num_splits() -> int:
    out = ctypes.c_int32(0)
    _check(load().eg_mla_default_num_splits(ctypes.byref(out)), "eg_mla_default_num_splits")
    return int(out.value)


def eg_mla_decode_workspace_size(dims: EgMlaDims, batch: int, num_splits: int = 0) -> int:
    n = load().eg_mla_decode_workspace_size(ctypes.byref(dims), batch, num_splits)
    if n == 0:
        raise EgMlaError(EG_MLA_ERR_UNSUPPORTED, "eg_mla_decode_workspace_size")
    return int(n)


def eg_mla_kv_bytes_per_token(dims: EgMlaDims, n_layers: int) -> int:
    out = ctypes.c_int64(0)
    _check(load().eg_mla_kv_bytes_per_token(ctypes.byref(dims), n_layers, ctypes.byref(out)),
           "eg_mla_kv_bytes_per_token")
    return int(out.value)


def eg_mla_append_latent(dims: EgMlaDims, c_pool, krope_pool, id_pool, c_new, krope_new, ids_new,
                         block_table, positions, dev_status=None, stream=None) -> None:
    code = load().eg_mla_append_latent(
        ctypes.byref(dims), _ptr(c_pool), _ptr(krope_pool), _ptr(id_pool), _ptr(c_new), _ptr(krope_new),
        _ptr(ids_new), _ptr(block_table), block_table.shape[1], _ptr(positions), positions.shape[0],
        c_pool.shape[0], _ptr(dev_status), _stream(stream))
    _check(code, "eg_mla_append_latent")


def eg_mla_decode(dims: EgMlaDims, q, c_pool, krope_pool, id_pool, block_table, seq_lens, max_seq_len,
                  gate_table, ln_gamma, ln_beta, w_uk, w_uv, out, workspace, num_splits=0,
                  dev_status=None, stream=None) -> None:
    code = load().eg_mla_decode(
        ctypes.byref(dims), _ptr(q), _ptr(c_pool), _ptr(krope_pool), _ptr(id_pool), _ptr(block_table),
        block_table.shape[1], _ptr(seq_lens), int(max_seq_len), seq_lens.shape[0], c_pool.shape[0],
        _ptr(gate_table), _ptr(ln_gamma), _ptr(ln_beta), _ptr(w_uk), _ptr(w_uv), _ptr(out), num_splits,
        _ptr(workspace), workspace.numel() * workspace.element_size(), _ptr(dev_status), _stream(stream))
    _check(code, "eg_mla_decode")


def _step_args(dims, c_pool, krope_pool, id_pool, c_new, krope_new, ids_new, positions, q, block_table, seq_lens,
               max_seq_len, gate_table, ln_gamma, ln_beta, w_uk, w_uv, out, workspace, num_splits, dev_status,
               stream):
    return (ctypes.byref(dims), _ptr(c_pool), _ptr(krope_pool), _ptr(id_pool), _ptr(c_new), _ptr(krope_new),
            _ptr(ids_new), _ptr(positions), _ptr(q), _ptr(block_table), block_table.shape[1], _ptr(seq_lens),
            int(max_seq_len), seq_lens.shape[0], c_pool.shape[0], _ptr(gate_table), _ptr(ln_gamma), _ptr(ln_beta),
            _ptr(w_uk), _ptr(w_uv), _ptr(out), num_splits, _ptr(workspace),
            workspace.numel() * workspace.element_size(), _ptr(dev_status), _stream(stream))


def eg_mla_step(dims: EgMlaDims, c_pool, krope_pool, id_pool, c_new, krope_new, ids_new, positions, q, block_table,
                seq_lens, max_seq_len, gate_table, ln_gamma, ln_beta, w_uk, w_uv, out, workspace, num_splits=0,
                dev_status=None, stream=None) -> None:
    """eg_mla_append_latent followed by eg_mla_decode, as one C call."""
    _check(load().eg_mla_step(*_step_args(dims, c_pool, krope_pool, id_pool, c_new, krope_new, ids_new, positions,
                                          q, block_table, seq_lens, max_seq_len, gate_table, ln_gamma, ln_beta,
                                          w_uk, w_uv, out, workspace, num_splits, dev_status, stream)),
           "eg_mla_step")


def eg_mla_decode_static(dims: EgMlaDims, q, c_pool, krope_pool, id_pool, block_table, seq_lens, max_seq_len,
                         gate_table, ln_gamma, ln_beta, w_uk, w_uv, out, num_splits=0,
                         dev_status=None, stream=None) -> None:
    """eg_mla_decode on the library's static scratch array (no workspace argument)."""
    code = load().eg_mla_decode_static(
        ctypes.byref(dims), _ptr(q), _ptr(c_pool), _ptr(krope_pool), _ptr(id_pool), _ptr(block_table),
        block_table.shape[1], _ptr(seq_lens), int(max_seq_len), seq_lens.shape[0], c_pool.shape[0],
        _ptr(gate_table), _ptr(ln_gamma), _ptr(ln_beta), _ptr(w_uk), _ptr(w_uv), _ptr(out), num_splits,
        _ptr(dev_status), _stream(stream))
    _check(code, "eg_mla_decode_static")


def make_layer_dims(n_embd: int, rope_theta: float = 10000.0, rms_eps: float = 0.0,
                    share_kv: bool = False) -> EgMlaLayerDims:
    """share_kv: a later layer of a layer group (its group's first layer projects
    and appends the shared c^KV, k^R; this one attends over the shared cache)."""
    return EgMlaLayerDims(n_embd, rope_theta, rms_eps, 1 if share_kv else 0)


def make_layer_weights(w_qkv_a, kv_norm_w, w_o, gate_table, ln_gamma, ln_beta, w_uk, w_uv) -> EgMlaLayerWeights:
    """w_qkv_a: the rows of W^Q stacked on those of W^{DKV,KR} ([nq + d_c + d_rope, E])."""
    return EgMlaLayerWeights(*[_ptr(t) for t in (w_qkv_a, kv_norm_w, w_o, gate_table, ln_gamma, ln_beta, w_uk, w_uv)])


def eg_mla_layer_workspace_size(dims: EgMlaDims, layer: EgMlaLayerDims, batch: int, num_splits: int = 0) -> int:
    n = load().eg_mla_layer_workspace_size(ctypes.byref(dims), ctypes.byref(layer), batch, num_splits)
    if n == 0:
        raise EgMlaError(EG_MLA_ERR_UNSUPPORTED, "eg_mla_layer_workspace_size")
    return int(n)


def eg_mla_layer_attn_offset(dims: EgMlaDims, layer: EgMlaLayerDims, batch: int, num_splits: int = 0) -> int:
    n = load().eg_mla_layer_attn_offset(ctypes.byref(dims), ctypes.byref(layer), batch, num_splits)
    if n == 0:
        raise EgMlaError(EG_MLA_ERR_UNSUPPORTED, "eg_mla_layer_attn_offset")
    return int(n)


def eg_mla_layer_decode(dims: EgMlaDims, layer: EgMlaLayerDims, weights: EgMlaLayerWeights, x, ids_new, positions,
                        c_pool, krope_pool, id_pool, block_table, seq_lens, max_seq_len, y, workspace,
                        num_splits=0, dev_status=None, stream=None) -> None:
    """One decode step through a whole attention layer (see include/egmla.h)."""
    code = load().eg_mla_layer_decode(
        ctypes.byref(dims), ctypes.byref(layer), ctypes.byref(weights), _ptr(x), _ptr(ids_new), _ptr(positions),
        _ptr(c_pool), _ptr(krope_pool), _ptr(id_pool), _ptr(block_table), block_table.shape[1], _ptr(seq_lens),
        int(max_seq_len), seq_lens.shape[0], c_pool.shape[0], _ptr(y), num_splits, _ptr(workspace),
        workspace.numel() * workspace.element_size(), _ptr(dev_status), _stream(stream))
    _check(code, "eg_mla_layer_decode")


def bind_step(dims: EgMlaDims, c_pool, krope_pool, id_pool, c_new, krope_new, ids_new, positions, q, block_table,
              seq_lens, max_seq_len, gate_table, ln_gamma, ln_beta, w_uk, w_uv, out, workspace, num_splits=0,
              dev_status=None, stream=None):
    """One decode step (eg_mla_step: append, then decode) with every argument
    converted once: returns a callable that issues the C call on `stream` with
    those pointers.  The tensors must stay alive and in place while the
    callable is used; a caller that reruns the same step every token saves the
    per-call argument marshalling."""
    fn = load().eg_mla_step
    args = _step_args(dims, c_pool, krope_pool, id_pool, c_new, krope_new, ids_new, positions, q, block_table,
                      seq_lens, max_seq_len, gate_table, ln_gamma, ln_beta, w_uk, w_uv, out, workspace, num_splits,
                      dev_status, stream)

    def step() -> None:
        rc = fn(*args)
        if rc != EG_MLA_OK:
            raise EgMlaError(rc, "eg_mla_step")

    step.keepalive = (dims, c_pool, krope_pool, id_pool, c_new, krope_new, ids_new, positions, q, block_table,
                      seq_lens, gate_table, ln_gamma, ln_beta, w_uk, w_uv, out, workspace, dev_status)
    return step


def eg_mla_decode_r0_workspace_size(dims: EgMlaDims, batch: int, max_pages_per_seq: int, num_pages: int) -> int:
    n = load().eg_mla_decode_r0_workspace_size(ctypes.byref(dims), int(batch), int(max_pages_per_seq),
                                               int(num_pages))
    if n == 0:
        raise EgMlaError(EG_MLA_ERR_UNSUPPORTED, "eg_mla_decode_r0_workspace_size")
    return int(n)


def eg_mla_decode_r0(dims: EgMlaDims, q, c_pool, krope_pool, id_pool, block_table, seq_lens, w_ukv, gate_r0,
                     ln_gamma, ln_beta, out, workspace, dev_status=None, stream=None) -> None:
    """Paper-literal (R0) gated decode: see include/egmla.h."""
    code = load().eg_mla_decode_r0(
        ctypes.byref(dims), _ptr(q), _ptr(c_pool), _ptr(krope_pool), _ptr(id_pool), _ptr(block_table),
        block_table.shape[1], _ptr(seq_lens), seq_lens.shape[0], c_pool.shape[0], _ptr(w_ukv), _ptr(gate_r0),
        _ptr(ln_gamma), _ptr(ln_beta), _ptr(out), _ptr(workspace), workspace.numel() * workspace.element_size(),
        _ptr(dev_status), _stream(stream))
    _check(code, "eg_mla_decode_r0")


def eg_mla_prefill_workspace_size(dims: EgMlaDims, batch: int, total_tokens: int) -> int:
    n = load().eg_mla_prefill_workspace_size(ctypes.byref(dims), int(batch), int(total_tokens))
    if n == 0 and total_tokens > 0:
        raise EgMlaError(EG_MLA_ERR_UNSUPPORTED, "eg_mla_prefill_workspace_size")
    return int(n)


def eg_mla_prefill(dims: EgMlaDims, q, c_new, krope_new, ids_new, cu_seqlens, max_seq_len, gate_table,
                   ln_gamma, ln_beta, w_uk, w_uv, out, workspace, c_pool=None, krope_pool=None, id_pool=None,
                   block_table=None, dev_status=None, stream=None) -> None:
    """Prompt processing (causal attention over packed prompts, cache write):
    see include/egmla.h.  Sizes are taken from the tensors: batch =
    len(cu_seqlens) - 1, total_tokens = q.shape[0]."""
    code = load().eg_mla_prefill(
        ctypes.byref(dims), _ptr(q), _ptr(c_new), _ptr(krope_new), _ptr(ids_new), _ptr(cu_seqlens),
        cu_seqlens.shape[0] - 1, q.shape[0], int(max_seq_len), _ptr(gate_table), _ptr(ln_gamma), _ptr(ln_beta),
        _ptr(w_uk), _ptr(w_uv), _ptr(out), _ptr(c_pool), _ptr(krope_pool), _ptr(id_pool), _ptr(block_table),
        block_table.shape[1] if block_table is not None else 0, c_pool.shape[0] if c_pool is not None else 0,
        _ptr(workspace), workspace.numel() * workspace.element_size(), _ptr(dev_status), _stream(stream))
    _check(code, "eg_mla_prefill")


def eg_mla_gate_table(dims: EgMlaDims, emb, w_ue, gate_table, dev_status=None, stream=None) -> None:
    """G = E W^UE^T for every vocabulary entry: emb [vocab, d_e], w_ue [d_c, d_e],
    gate_table [vocab, d_c], all bf16 (see include/egmla.h)."""
    _check(load().eg_mla_gate_table(ctypes.byref(dims), emb.shape[1], _ptr(emb), _ptr(w_ue), _ptr(gate_table),
                                    _ptr(dev_status), _stream(stream)), "eg_mla_gate_table")


def eg_mla_debug_linear(w, x, out, dev_status=None, stream=None) -> None:
    """out[:, :n_out] = x @ w.T through the layer's projection GEMM (w [n_out, k],
    x [batch, k] bf16; out fp32 or bf16 with out.shape[1] >= n_out)."""
    n_out, k = w.shape
    _check(load().eg_mla_debug_linear(_ptr(w), n_out, k, _ptr(x), x.shape[0], _ptr(out), out.shape[1],
                                      1 if out.dtype == torch.float32 else 0, _ptr(dev_status), _stream(stream)),
           "eg_mla_debug_linear")


def eg_mla_debug_linear_plan(n_out: int, k: int, batch: int) -> dict:
    """The projection GEMM's launch shape for these sizes (no launch)."""
    c, st, m = ctypes.c_int32(0), ctypes.c_int32(0), ctypes.c_int32(0)
    _check(load().eg_mla_debug_linear_plan(n_out, k, batch, ctypes.byref(c), ctypes.byref(st), ctypes.byref(m)),
           "eg_mla_debug_linear_plan")
    return {"cluster": int(c.value), "stages": int(st.value), "max_clusters": int(m.value)}


def eg_mla_debug_gather(dims: EgMlaDims, c_pool, krope_pool, id_pool, block_table, seq_lens, max_seq_len,
                        gate_table, c_out, kr_out, ids_out, g_out, workspace, num_splits=0,
                        dev_status=None, stream=None) -> None:
    code = load().eg_mla_debug_gather(
        ctypes.byref(dims), _ptr(c_pool), _ptr(krope_pool), _ptr(id_pool), _ptr(block_table),
        block_table.shape[1], _ptr(seq_lens), int(max_seq_len), seq_lens.shape[0], c_pool.shape[0],
        _ptr(gate_table), _ptr(c_out), _ptr(kr_out), _ptr(ids_out), _ptr(g_out), num_splits,
        _ptr(workspace), workspace.numel() * workspace.element_size(), _ptr(dev_status), _stream(stream))
    _check(code, "eg_mla_debug_gather")


def eg_mla_profile_begin(max_launches: int) -> None:
    _check(load().eg_mla_profile_begin(max_launches), "eg_mla_profile_begin")


def eg_mla_profile_end():
    """(summed decode-kernel milliseconds, launches timed)."""
    ms = ctypes.c_double(0)
    n = ctypes.c_int32(0)
    _check(load().eg_mla_profile_end(ctypes.byref(ms), ctypes.byref(n)), "eg_mla_profile_end")
    return float(ms.value), int(n.value)


def eg_mla_debug_set_trace(buf: Optional[torch.Tensor], ctas: int = 0) -> None:
    """Set (or clear, with None) the decode kernel's pipeline trace buffer."""
    if buf is None:
        _check(load().eg_mla_debug_set_trace(None, 0, 0), "eg_mla_debug_set_trace")
        return
    _check(load().eg_mla_debug_set_trace(_ptr(buf), buf.numel() * buf.element_size(), ctas),
           "eg_mla_debug_set_trace")


def eg_mla_debug_set_fault(cta: int = -1, tile: int = 0, wait_limit_ns: int = 0) -> None:
    """Withhold the page copy of tile `tile` of CTA `cta` in later decode calls and
    lower their wait limit (cta < 0: back to normal)."""
    _check(load().eg_mla_debug_set_fault(cta, tile, wait_limit_ns), "eg_mla_debug_set_fault")

"""Device-side plumbing: upload a synthetic decode step to HBM and run it
through the C ABI (append of the new token, then decode).

PyTorch only allocates device memory and provides the stream here; the work
itself is done by libegmla's kernels.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np
import torch

from . import _lib
from .synth import Case


def to_device_array(a: np.ndarray, dtype: str, device) -> torch.Tensor:
    """Stored bits -> device tensor of the model dtype (bf16 from uint16 bits)."""
    if dtype == "bf16" and a.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(device)
    if a.dtype == np.int32:
        return torch.from_numpy(np.ascontiguousarray(a)).to(device)
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device)


def bf16_tensor_to_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


@dataclasses.dataclass
class DeviceCase:
    dims: _lib.EgMlaDims
    dtype: str
    c_pool: torch.Tensor
    kr_pool: torch.Tensor
    id_pool: torch.Tensor
    block_table: torch.Tensor
    seq_lens: torch.Tensor
    positions: torch.Tensor
    c_new: torch.Tensor
    kr_new: torch.Tensor
    ids_new: torch.Tensor
    q: torch.Tensor
    gate_table: torch.Tensor
    ln_gamma: torch.Tensor
    ln_beta: torch.Tensor
    w_uk: torch.Tensor
    w_uv: torch.Tensor
    out: torch.Tensor
    workspace: torch.Tensor
    status: torch.Tensor
    max_seq_len: int
    num_splits: int

    @property
    def batch(self) -> int:
        return int(self.seq_lens.shape[0])

    def append(self, stream=None) -> None:
        _lib.eg_mla_append_latent(self.dims, self.c_pool, self.kr_pool, self.id_pool, self.c_new, self.kr_new,
                                  self.ids_new, self.block_table, self.positions, self.status, stream)

    def decode(self, stream=None, out: Optional[torch.Tensor] = None) -> torch.Tensor:
        o = self.out if out is None else out
        _lib.eg_mla_decode(self.dims, self.q, self.c_pool, self.kr_pool, self.id_pool, self.block_table,
                           self.seq_lens, self.max_seq_len, self.gate_table, self.ln_gamma, self.ln_beta,
                           self.w_uk, self.w_uv, o, self.workspace, self.num_splits, self.status, stream)
        return o

    def step(self, stream=None, out: Optional[torch.Tensor] = None) -> torch.Tensor:
        """One decode step (eg_mla_step): append the new token, then attend over
        the cache."""
        o = self.out if out is None else out
        _lib.eg_mla_step(self.dims, self.c_pool, self.kr_pool, self.id_pool, self.c_new, self.kr_new, self.ids_new,
                         self.positions, self.q, self.block_table, self.seq_lens, self.max_seq_len, self.gate_table,
                         self.ln_gamma, self.ln_beta, self.w_uk, self.w_uv, o, self.workspace, self.num_splits,
                         self.status, stream)
        return o

    def bind(self, stream=None):
        """step() with its C-ABI arguments converted once (see _lib.bind_step)."""
        return _lib.bind_step(self.dims, self.c_pool, self.kr_pool, self.id_pool, self.c_new, self.kr_new,
                              self.ids_new, self.positions, self.q, self.block_table, self.seq_lens,
                              self.max_seq_len, self.gate_table, self.ln_gamma, self.ln_beta, self.w_uk, self.w_uv,
                              self.out, self.workspace, self.num_splits, self.status, stream)

    def read_status(self) -> int:
        return int(self.status.item())


def dims_of(case: Case) -> _lib.EgMlaDims:
    d = case.dims
    return _lib.make_dims(d.num_heads, d.d_nope, d.d_rope, d.d_v, d.d_c, d.vocab, dtype=d.dtype, gate=d.gate,
                          page_size=d.page_size, softmax_scale=d.softmax_scale, ln_eps=d.ln_eps,
                          gate_op=getattr(d, "gate_op", "mul_ln"))


def upload(case: Case, device="cuda", num_splits: int = 0) -> DeviceCase:
    d = case.dims
    dt = d.dtype
    dims = dims_of(case)
    B = case.batch
    ws_bytes = _lib.eg_mla_decode_workspace_size(dims, B, num_splits)
    out_dtype = torch.bfloat16 if dt == "bf16" else torch.float32
    return DeviceCase(
        dims=dims, dtype=dt,
        c_pool=to_device_array(case.c_pool, dt, device),
        kr_pool=to_device_array(case.kr_pool, dt, device),
        id_pool=to_device_array(case.id_pool, dt, device),
        block_table=to_device_array(case.block_table, dt, device),
        seq_lens=to_device_array(case.seq_lens, dt, device),
        positions=to_device_array(case.positions(), dt, device),
        c_new=to_device_array(case.c_new, dt, device),
        kr_new=to_device_array(case.kr_new, dt, device),
        ids_new=to_device_array(case.ids_new, dt, device),
        q=to_device_array(case.q, dt, device),
        gate_table=to_device_array(case.gate_table, dt, device),
        ln_gamma=torch.from_numpy(case.ln_gamma.astype(np.float32)).to(device),
        ln_beta=torch.from_numpy(case.ln_beta.astype(np.float32)).to(device),
        w_uk=to_device_array(case.w_uk, dt, device),
        w_uv=to_device_array(case.w_uv, dt, device),
        out=torch.empty((B, d.num_heads, d.d_v), dtype=out_dtype, device=device),
        workspace=torch.empty(ws_bytes, dtype=torch.uint8, device=device),
        status=torch.zeros(1, dtype=torch.int32, device=device),
        max_seq_len=int(case.seq_lens.max()) if B else 0,
        num_splits=num_splits,
    )


def clone_case(dc: DeviceCase, share=("workspace", "status")) -> DeviceCase:
    """A copy of `dc` in distinct device memory (same values), sharing the
    fields named in `share` (e.g. one workspace for units run in sequence)."""
    fields = {}
    for f in dataclasses.fields(dc):
        v = getattr(dc, f.name)
        fields[f.name] = v.clone() if isinstance(v, torch.Tensor) and f.name not in share else v
    return DeviceCase(**fields)


# inputs that change from one decode step to the next
STEP_INPUTS = ("q", "c_new", "kr_new", "ids_new", "positions", "seq_lens")


def pack_step_inputs(dc: DeviceCase, names=STEP_INPUTS):
    """Move the per-step inputs of `dc` into one device buffer (each a view at a
    256-byte aligned offset, so the C ABI's 16-byte alignment rules hold) and
    return (pinned host buffer, device buffer) with the same bytes: a step's
    host-to-device traffic is then a single copy instead of one per tensor."""
    layout, off = [], 0
    for n in names:
        t = getattr(dc, n)
        nbytes = t.numel() * t.element_size()
        layout.append((n, off, nbytes))
        off = (off + nbytes + 255) // 256 * 256
    dev = torch.empty(off, dtype=torch.uint8, device=dc.q.device)
    host = torch.zeros(off, dtype=torch.uint8).pin_memory()
    for n, o, nbytes in layout:
        t = getattr(dc, n).contiguous()
        view = dev[o:o + nbytes].view(t.dtype).view(t.shape)
        view.copy_(t)
        host[o:o + nbytes].copy_(t.cpu().view(torch.uint8).reshape(-1))
        setattr(dc, n, view)
    return host, dev


def output_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


@dataclasses.dataclass
class DeviceLayer:
    """One attention layer's decode step on the device: the cache and decode
    inputs of ``dc`` plus the hidden state, the projection weights, the output
    and the layer workspace."""
    dc: DeviceCase
    layer_dims: _lib.EgMlaLayerDims
    x: torch.Tensor
    w_qkv_a: torch.Tensor       # [W^Q ; W^{DKV,KR}] stacked by rows
    kv_norm_w: torch.Tensor
    w_o: torch.Tensor
    y: torch.Tensor
    workspace: torch.Tensor

    def weights(self) -> _lib.EgMlaLayerWeights:
        dc = self.dc
        return _lib.make_layer_weights(self.w_qkv_a, self.kv_norm_w, self.w_o, dc.gate_table, dc.ln_gamma,
                                       dc.ln_beta, dc.w_uk, dc.w_uv)

    def step(self, stream=None) -> torch.Tensor:
        """x -> y: projections, kv_norm and RoPE, append, decode, output projection."""
        dc = self.dc
        _lib.eg_mla_layer_decode(dc.dims, self.layer_dims, self.weights(), self.x, dc.ids_new, dc.positions,
                                 dc.c_pool, dc.kr_pool, dc.id_pool, dc.block_table, dc.seq_lens, dc.max_seq_len,
                                 self.y, self.workspace, dc.num_splits, dc.status, stream)
        return self.y

    def attn_output(self) -> torch.Tensor:
        """The last step's attention output u [B, H, d_v] (bf16), read from where
        eg_mla_layer_decode leaves it in the workspace."""
        dc = self.dc
        off = _lib.eg_mla_layer_attn_offset(dc.dims, self.layer_dims, dc.batch, dc.num_splits)
        n = dc.batch * dc.dims.num_heads * dc.dims.d_v * 2
        return self.workspace[off:off + n].view(torch.bfloat16).view(dc.batch, dc.dims.num_heads, dc.dims.d_v)


def upload_layer(lc, device="cuda", num_splits: int = 0) -> DeviceLayer:
    """A synth.LayerCase on the device (bf16)."""
    dc = upload(lc.case, device=device, num_splits=num_splits)
    dt = lc.case.dims.dtype
    ld = _lib.make_layer_dims(lc.n_embd, lc.rope_theta, lc.rms_eps)
    ws = _lib.eg_mla_layer_workspace_size(dc.dims, ld, dc.batch, num_splits)
    return DeviceLayer(
        dc=dc, layer_dims=ld,
        x=to_device_array(lc.x, dt, device),
        w_qkv_a=to_device_array(np.concatenate([lc.w_q, lc.w_kv_a], axis=0), dt, device),
        kv_norm_w=to_device_array(lc.kv_norm_w, dt, device),
        w_o=to_device_array(lc.w_o, dt, device),
        y=torch.empty((dc.batch, lc.n_embd), dtype=torch.bfloat16, device=device),
        workspace=torch.empty(ws, dtype=torch.uint8, device=device))


def clone_layer(dl: DeviceLayer, share=("workspace", "status")) -> DeviceLayer:
    """Another layer of the same shape: its own cache and weights (same values),
    its own output; the decode and layer workspaces and the status word shared
    (layers run one after another on one stream), and whatever else of the
    cache ``share`` names (a layer group shares its pools and block table)."""
    return DeviceLayer(dc=clone_case(dl.dc, share=share), layer_dims=dl.layer_dims, x=dl.x.clone(),
                       w_qkv_a=dl.w_qkv_a.clone(),
                       kv_norm_w=dl.kv_norm_w.clone(), w_o=dl.w_o.clone(),
                       y=torch.empty_like(dl.y), workspace=dl.workspace)


# --------------------------------------------------------------------------
# prompt processing (prefill)
# --------------------------------------------------------------------------
@dataclasses.dataclass
class DevicePrefill:
    dims: _lib.EgMlaDims
    q: torch.Tensor
    c: torch.Tensor
    kr: torch.Tensor
    ids: torch.Tensor
    cu_seqlens: torch.Tensor
    gate_table: torch.Tensor
    ln_gamma: torch.Tensor
    ln_beta: torch.Tensor
    w_uk: torch.Tensor
    w_uv: torch.Tensor
    c_pool: torch.Tensor
    kr_pool: torch.Tensor
    id_pool: torch.Tensor
    block_table: torch.Tensor
    out: torch.Tensor
    workspace: torch.Tensor
    status: torch.Tensor
    max_seq_len: int

    def run(self, stream=None, write_cache: bool = True) -> torch.Tensor:
        """eg_mla_prefill over the packed prompts (and the cache write)."""
        pools = (self.c_pool, self.kr_pool, self.id_pool, self.block_table) if write_cache else (None,) * 4
        _lib.eg_mla_prefill(self.dims, self.q, self.c, self.kr, self.ids, self.cu_seqlens, self.max_seq_len,
                            self.gate_table, self.ln_gamma, self.ln_beta, self.w_uk, self.w_uv, self.out,
                            self.workspace, *pools, dev_status=self.status, stream=stream)
        return self.out

    def read_status(self) -> int:
        return int(self.status.item())


def upload_prefill(pc, device="cuda") -> DevicePrefill:
    d = pc.dims
    dt = d.dtype
    dims = dims_of(pc)
    T = pc.total_tokens
    return DevicePrefill(
        dims=dims,
        q=to_device_array(pc.q, dt, device),
        c=to_device_array(pc.c, dt, device),
        kr=to_device_array(pc.kr, dt, device),
        ids=to_device_array(pc.ids, dt, device),
        cu_seqlens=to_device_array(pc.cu_seqlens, dt, device),
        gate_table=to_device_array(pc.gate_table, dt, device),
        ln_gamma=torch.from_numpy(pc.ln_gamma.astype(np.float32)).to(device),
        ln_beta=torch.from_numpy(pc.ln_beta.astype(np.float32)).to(device),
        w_uk=to_device_array(pc.w_uk, dt, device),
        w_uv=to_device_array(pc.w_uv, dt, device),
        c_pool=to_device_array(pc.c_pool, dt, device),
        kr_pool=to_device_array(pc.kr_pool, dt, device),
        id_pool=to_device_array(pc.id_pool, dt, device),
        block_table=to_device_array(pc.block_table, dt, device),
        out=torch.empty((T, d.num_heads, d.d_v), dtype=torch.bfloat16, device=device),
        workspace=torch.empty(max(_lib.eg_mla_prefill_workspace_size(dims, pc.batch, T), 1), dtype=torch.uint8,
                              device=device),
        status=torch.zeros(1, dtype=torch.int32, device=device),
        max_seq_len=int(pc.seq_lens.max()) if pc.batch else 0,
    )

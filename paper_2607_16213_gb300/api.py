"""Torch-facing helpers around the C ABI: allocate device tensors and workspaces with torch,
then call selkv_compress / selkv_decode_attn.  No arithmetic of the method happens here."""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Optional, Sequence

import torch

from . import _binding as B

_TORCH_DTYPE = {B.SELKV_BF16: torch.bfloat16, B.SELKV_FP32: torch.float32}
_DTYPE_CODE = {"bf16": B.SELKV_BF16, "fp32": B.SELKV_FP32}


def dtype_code(name: str) -> int:
    return _DTYPE_CODE[name]


def torch_dtype(code: int) -> torch.dtype:
    return _TORCH_DTYPE[code]


def make_shape(dtype: str, batch: int, num_q_heads: int, num_kv_heads: int, head_dim: int,
               obs_window: int, n_cap: int, m_cap: int) -> B.selkv_shape:
    return B.selkv_shape(_DTYPE_CODE[dtype], batch, num_q_heads, num_kv_heads, head_dim,
                         obs_window, n_cap, m_cap)


def capacity(n_max: int, rho: float, extra: int = 0, align: int = 64) -> int:
    """A row capacity that holds floor(rho * n_max) compressed rows plus `extra` appended rows."""
    need = int(math.floor(float(rho) * float(n_max))) + extra
    return max(align, ((need + align - 1) // align) * align)


class Workspace:
    """A zero-initialised device workspace of at least `nbytes` (256-byte aligned)."""

    def __init__(self, nbytes: int, device="cuda", stream=None):
        self.nbytes = max(256, int(nbytes))
        self.buf = torch.empty(self.nbytes, dtype=torch.uint8, device=device)
        B.check(B.selkv_workspace_init(self.buf, self.nbytes, stream), "selkv_workspace_init")

    def ptr(self) -> int:
        return self.buf.data_ptr()

    def errors(self, stream=None) -> int:
        st, flags = B.selkv_workspace_error(self.buf, stream)
        return flags


@dataclass
class CompressedCache:
    shape: B.selkv_shape
    K_c: torch.Tensor
    V_c: torch.Tensor
    bias: torch.Tensor
    lengths: torch.Tensor
    debug: dict = field(default_factory=dict)


def alloc_compressed(shape: B.selkv_shape, device="cuda") -> CompressedCache:
    dt = _TORCH_DTYPE[shape.dtype]
    Bn, H, m, d = shape.batch, shape.num_kv_heads, shape.m_cap, shape.head_dim
    return CompressedCache(shape=shape,
                           K_c=torch.zeros((Bn, H, m, d), dtype=dt, device=device),
                           V_c=torch.zeros((Bn, H, m, d), dtype=dt, device=device),
                           bias=torch.zeros((Bn, H, m), dtype=torch.float32, device=device),
                           lengths=torch.zeros((Bn,), dtype=torch.int32, device=device))


def alloc_debug(shape: B.selkv_shape, device="cuda", per_head: bool = False) -> dict:
    """Debug outputs of selkv_compress (kept_idx is per KV head in the per-head mode)."""
    Bn, H, n, m = shape.batch, shape.num_kv_heads, shape.n_cap, shape.m_cap
    return dict(
        attn=torch.zeros((Bn, H, n), dtype=torch.float32, device=device),
        score=torch.zeros((Bn, H, n), dtype=torch.float32, device=device),
        topk=torch.zeros((Bn, H, n), dtype=torch.uint8, device=device),
        kept_idx=torch.full((Bn, H, m) if per_head else (Bn, m), -1, dtype=torch.int32, device=device),
        target=torch.full((Bn, H, n), -7, dtype=torch.int32, device=device),
        gate=torch.zeros((Bn, H, n), dtype=torch.float32, device=device),
        decision=torch.full((Bn, H, n), 9, dtype=torch.uint8, device=device),
        ratio=torch.zeros((Bn, H, m), dtype=torch.float32, device=device),
    )


def compress(shape: B.selkv_shape, n_len: Sequence[int], rho: float, K: torch.Tensor,
             V: torch.Tensor, Q_obs: torch.Tensor, params: Optional[B.selkv_params] = None,
             out: Optional[CompressedCache] = None, debug: bool = False,
             workspace: Optional[Workspace] = None, stream=None) -> CompressedCache:
    """selkv_compress on device tensors; returns the compressed cache (and debug outputs)."""
    params = params or B.selkv_params.defaults()
    out = out or alloc_compressed(shape, K.device)
    dbg = alloc_debug(shape, K.device, per_head=params.select_mode == B.SELKV_SELECT_PER_HEAD) if debug else None
    ws = workspace or Workspace(B.selkv_compress_workspace_size(shape), K.device, stream)
    st = B.selkv_compress(shape, n_len, rho, params, K, V, Q_obs, out.K_c, out.V_c, out.bias,
                          out.lengths, dbg, ws.buf, ws.nbytes, stream)
    B.check(st, "selkv_compress")
    if dbg is not None:
        out.debug = dbg
    return out


def decode(cache: CompressedCache, q: torch.Tensor, k_new: Optional[torch.Tensor] = None,
           v_new: Optional[torch.Tensor] = None, use_bias: bool = True,
           out: Optional[torch.Tensor] = None, workspace: Optional[Workspace] = None,
           stream=None) -> torch.Tensor:
    """selkv_decode_attn over a compressed cache (optionally appending k_new / v_new)."""
    shape = cache.shape
    out = out if out is not None else torch.empty_like(q)
    ws = workspace or Workspace(B.selkv_decode_workspace_size(shape), q.device, stream)
    st = B.selkv_decode_attn(shape, q, cache.K_c, cache.V_c, cache.bias if use_bias else None,
                             cache.lengths, k_new, v_new, out, ws.buf, ws.nbytes, stream)
    B.check(st, "selkv_decode_attn")
    return out

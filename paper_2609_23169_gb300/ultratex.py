"""Python binding of libultratex.so (ctypes; argument marshalling only).

Every function here has the name of the C entry point it wraps and does
nothing but check Python-side arguments, allocate outputs with torch when the
caller did not pass them, and call the library on the current CUDA stream.
There is no fallback: if the library is missing or a call fails, it raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "lib", "libultratex.so")

UT_OK, UT_ERR_INVALID_ARG, UT_ERR_UNSUPPORTED, UT_ERR_CUDA, UT_ERR_TIMEOUT, UT_ERR_CAPACITY = range(6)
UT_BF16, UT_F32 = 0, 1
UT_BG_KEEP, UT_BG_ZERO, UT_BG_FILL = 0, 1, 2
UT_MASK_TOPK, UT_MASK_BITMAP = 0, 1

EXPORTS = (
    "ut_strerror", "ut_topk_count", "ut_fg_compact_workspace_size", "ut_fg_compact", "ut_fg_scatter",
    "ut_block_mask_workspace_size", "ut_block_mask", "ut_bsattn_fwd", "ut_bsattn_bwd_workspace_size",
    "ut_bsattn_bwd", "ut_fg_compact_noalloc", "ut_fg_euler_update", "ut_fg_euler_update_gather", "ut_fg_composite",
    "ut_fg_gather_rope", "ut_fg_scatter_rope", "ut_fg_mask_from_alpha", "ut_device_accessible",
)


class UtError(RuntimeError):
    def __init__(self, fn: str, status: int, msg: str):
        super().__init__(f"{fn} failed: {msg} (status {status})")
        self.status = status


class AttnShape(ctypes.Structure):
    _fields_ = [("n_tokens", ctypes.c_int64), ("n_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("block", ctypes.c_int32), ("dtype", ctypes.c_int32), ("row_stride", ctypes.c_int64),
                ("block_k", ctypes.c_int32)]


class Rope(ctypes.Structure):
    """ut_rope: tokens per image side, head dimensions of the image / y / x axes, frequency base, text prefix."""
    _fields_ = [("side", ctypes.c_int32), ("axes", ctypes.c_int32 * 3), ("theta", ctypes.c_float),
                ("prefix", ctypes.c_int32)]


def rope_config(side: int, axes=(16, 56, 56), theta: float = 10000.0, prefix: int = 0) -> Rope:
    return Rope(int(side), (ctypes.c_int32 * 3)(*axes), float(theta), int(prefix))


_lib = None
_vp, _i32, _i64, _sz, _dbl, _flt = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t,
                                     ctypes.c_double, ctypes.c_float)
_ptrs = ctypes.POINTER(ctypes.c_void_p)


def lib() -> ctypes.CDLL:
    """Load libultratex.so (built by __graft_entry__.build()); raise if absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
    L = ctypes.CDLL(LIB_PATH)
    L.ut_strerror.restype = ctypes.c_char_p
    L.ut_strerror.argtypes = [_i32]
    L.ut_topk_count.restype = _i32
    L.ut_topk_count.argtypes = [_dbl, _i64]
    L.ut_fg_compact_workspace_size.restype = _sz
    L.ut_fg_compact_workspace_size.argtypes = [_i64]
    L.ut_fg_compact.restype = _i32
    L.ut_fg_compact.argtypes = [_vp, _i64, _i32, _ptrs, _ptrs, _i64, _i64, _vp, _vp, _vp, _sz, _vp, _vp]
    L.ut_fg_scatter.restype = _i32
    L.ut_fg_scatter.argtypes = [_vp, _i64, _i32, _ptrs, _ptrs, _i64, _i32, _vp, _i64, _vp]
    L.ut_block_mask_workspace_size.restype = _sz
    L.ut_block_mask_workspace_size.argtypes = [ctypes.POINTER(AttnShape), _i32]
    L.ut_block_mask.restype = _i32
    L.ut_block_mask.argtypes = [ctypes.POINTER(AttnShape), _i32, _vp, _vp, _dbl, _vp, _vp, _vp, _i64, _vp, _vp,
                                _vp, _sz, _vp, _vp]
    L.ut_bsattn_fwd.restype = _i32
    L.ut_bsattn_fwd.argtypes = [ctypes.POINTER(AttnShape), _vp, _vp, _vp, _vp, _vp, _flt, _vp, _vp, _vp, _vp]
    L.ut_bsattn_bwd_workspace_size.restype = _sz
    L.ut_bsattn_bwd_workspace_size.argtypes = [ctypes.POINTER(AttnShape)]
    L.ut_bsattn_bwd.restype = _i32
    L.ut_bsattn_bwd.argtypes = [ctypes.POINTER(AttnShape), _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _flt,
                                _vp, _vp, _vp, _vp, _sz, _vp, _vp]
    L.ut_fg_euler_update.restype = _i32
    L.ut_fg_euler_update.argtypes = [_vp, _i64, _vp, _vp, _i64, _i32, _i32, _flt, _vp, _vp]
    L.ut_fg_euler_update_gather.restype = _i32
    L.ut_fg_euler_update_gather.argtypes = [_vp, _i64, _vp, _vp, _vp, _i64, _i32, _i32, _flt, _vp, _vp]
    L.ut_fg_composite.restype = _i32
    L.ut_fg_composite.argtypes = [_vp, _i64, _vp, _vp, _i64, _i64, _vp]
    L.ut_fg_gather_rope.restype = _i32
    L.ut_fg_gather_rope.argtypes = [_vp, _i64, _i32, _ptrs, _ptrs, _i64, _i32, _i32, _i32, ctypes.POINTER(Rope), _vp]
    L.ut_fg_scatter_rope.restype = _i32
    L.ut_fg_scatter_rope.argtypes = [_vp, _i64, _i32, _ptrs, _ptrs, _i64, _i32, _i32, _i32, ctypes.POINTER(Rope),
                                     _i32, _vp]
    L.ut_fg_mask_from_alpha.restype = _i32
    L.ut_fg_mask_from_alpha.argtypes = [_vp, _i32, _i32, _i32, _i32, _i32, _i32, _vp, _vp]
    L.ut_device_accessible.restype = _i32
    L.ut_device_accessible.argtypes = [_vp]
    _lib = L
    return L


def _check(fn: str, st: int) -> None:
    if st != UT_OK:
        raise UtError(fn, st, lib().ut_strerror(st).decode())


def _p(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream() -> int:
    return torch.cuda.current_stream().cuda_stream


def _ptr_array(ts: Sequence[torch.Tensor]):
    return (ctypes.c_void_p * len(ts))(*[t.data_ptr() for t in ts])


def _row_bytes(ts: Sequence[torch.Tensor], min_rows: int, what: str) -> int:
    """Common row size of a list of row-major tensors with at least min_rows rows.

    The C entry points take one row size for the whole list, so every tensor
    must share it; a mismatch would make the kernels read or write past a
    smaller tensor."""
    if len(ts) == 0:
        raise ValueError(f"{what} is empty")
    sizes = set()
    for t in ts:
        if not t.is_contiguous():
            raise ValueError(f"{what}: tensors must be contiguous")
        if t.shape[0] < min_rows:
            raise ValueError(f"{what}: a tensor has {t.shape[0]} rows, fewer than {min_rows}")
        sizes.add((t.numel() // max(1, t.shape[0])) * t.element_size() if t.shape[0] else -1)
    sizes.discard(-1)
    if len(sizes) > 1:
        raise ValueError(f"{what}: tensors differ in row size {sorted(sizes)}; one call per row size")
    return sizes.pop() if sizes else 16


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return UT_BF16
    if t.dtype == torch.float32:
        return UT_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def attn_shape(x: torch.Tensor, block: int, block_k: int = 0) -> AttnShape:
    """Shape of a token-major [N, H, d] tensor (rows may be padded: stride(0) >= H*d);
    query blocks of `block` rows, key blocks of `block_k` rows (0: same)."""
    N, H, d = x.shape
    assert x.stride(2) == 1 and x.stride(1) == d, "heads must be contiguous within a token row"
    return AttnShape(N, H, d, block, _dtype_code(x), x.stride(0), block_k)


def device_accessible(t: torch.Tensor) -> bool:
    """True if the library's kernels can address the tensor's storage directly
    (device memory, or host memory mapped into the device's address space)."""
    return bool(lib().ut_device_accessible(_p(t)))


def status_word(device=None) -> torch.Tensor:
    return torch.zeros(1, dtype=torch.int32, device=device or "cuda")


def check_status(st: torch.Tensor) -> None:
    v = int(st.item())
    if v != UT_OK:
        raise UtError("device", v, lib().ut_strerror(v).decode())


# ----------------------------------------------------------------- entry points
def ut_topk_count(rho: float, n_k: int) -> int:
    return int(lib().ut_topk_count(float(rho), int(n_k)))


def ut_fg_compact(mask: torch.Tensor, srcs: Sequence[torch.Tensor], capacity: Optional[int] = None,
                  outs: Optional[Sequence[torch.Tensor]] = None, idx: Optional[torch.Tensor] = None,
                  n_out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                  status: Optional[torch.Tensor] = None):
    """Background Token Dropping.  Returns (idx [capacity] i32, n_out [1] i32, outs)."""
    T = mask.shape[0]
    row_bytes = _row_bytes(srcs, T, "srcs")
    cap = T if capacity is None else int(capacity)
    dev = mask.device
    if outs is None:
        outs = [torch.empty((cap,) + tuple(s.shape[1:]), dtype=s.dtype, device=dev) for s in srcs]
    if len(outs) != len(srcs) or _row_bytes(outs, cap, "outs") != row_bytes:
        raise ValueError("outs must match srcs row for row")
    if idx is not None and idx.numel() < cap:
        raise ValueError("idx holds fewer than capacity entries")
    if idx is None:
        idx = torch.empty(max(cap, 1), dtype=torch.int32, device=dev)
    if n_out is None:
        n_out = torch.empty(1, dtype=torch.int32, device=dev)
    elif n_out.device.type != "cuda" and not device_accessible(n_out):
        raise ValueError("n_out must be device memory or host memory the device can address (pinned)")
    L = lib()
    wsb = L.ut_fg_compact_workspace_size(T)
    if ws is None:
        ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device=dev)
    st = L.ut_fg_compact(_p(mask), T, len(srcs), _ptr_array(srcs), _ptr_array(outs), row_bytes, cap, _p(idx),
                         _p(n_out), _p(ws), ws.numel(), _p(status), _stream())
    _check("ut_fg_compact", st)
    return idx, n_out, list(outs)


def ut_fg_scatter(idx: torch.Tensor, n: int, srcs: Sequence[torch.Tensor], dsts: Sequence[torch.Tensor],
                  bg_mode: int = UT_BG_KEEP, fill_row: Optional[torch.Tensor] = None) -> None:
    """dst[idx[i]] = src[i] for i < n; background rows per bg_mode."""
    T = dsts[0].shape[0]
    row_bytes = _row_bytes(dsts, T, "dsts")
    if len(srcs) != len(dsts) or _row_bytes(srcs, int(n), "srcs") != row_bytes:
        raise ValueError("srcs must match dsts row for row")
    if fill_row is not None and fill_row.numel() * fill_row.element_size() != row_bytes:
        raise ValueError("fill_row must hold exactly one row")
    if idx.numel() < int(n):
        raise ValueError("idx holds fewer than n entries")
    st = lib().ut_fg_scatter(_p(idx), int(n), len(srcs), _ptr_array(srcs), _ptr_array(dsts), row_bytes, bg_mode,
                             _p(fill_row), T, _stream())
    _check("ut_fg_scatter", st)


def ut_fg_mask_from_alpha(alpha: torch.Tensor, factor: int = 16, radius: int = 1, threshold: int = 0,
                          out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Canvas mask [(2V + 1) * h * w] uint8 from alpha [V + 1, height, width] uint8 (views, then reference)."""
    if alpha.dtype != torch.uint8 or alpha.dim() != 3 or not alpha.is_contiguous():
        raise ValueError("alpha must be a contiguous [V + 1, height, width] uint8 tensor")
    V = alpha.shape[0] - 1
    H, W = alpha.shape[1], alpha.shape[2]
    n = (2 * V + 1) * (H // max(factor, 1)) * (W // max(factor, 1))
    if out is None:
        out = torch.empty(max(n, 1), dtype=torch.uint8, device=alpha.device)
    elif out.numel() < n or out.dtype != torch.uint8:
        raise ValueError("out must hold (2V + 1) * (height/factor) * (width/factor) uint8")
    st = lib().ut_fg_mask_from_alpha(_p(alpha), V, H, W, factor, radius, threshold, _p(out), _stream())
    _check("ut_fg_mask_from_alpha", st)
    return out[:n]


def _rope_dims(ts: Sequence[torch.Tensor]):
    t0 = ts[0]
    if t0.dim() != 3 or t0.dtype not in (torch.bfloat16, torch.float32):
        raise ValueError("RoPE tensors are [rows, heads, head_dim] bf16 or fp32")
    for t in ts:
        if t.dim() != 3 or t.shape[1:] != t0.shape[1:] or t.dtype != t0.dtype or not t.is_contiguous():
            raise ValueError("RoPE tensors must share heads, head_dim and dtype, contiguous")
    return t0.shape[1], t0.shape[2], (UT_BF16 if t0.dtype == torch.bfloat16 else UT_F32)


def ut_fg_gather_rope(idx: torch.Tensor, n: int, srcs: Sequence[torch.Tensor], rope: Rope,
                      dsts: Optional[Sequence[torch.Tensor]] = None):
    """Rotated gather: dst[i] = R(idx[i]) src[idx[i]] for i < n.  Returns the dst list."""
    H, d, dtype = _rope_dims(srcs)
    if dsts is None:
        dsts = [torch.empty((max(int(n), 1), H, d), dtype=s.dtype, device=s.device) for s in srcs]
    _rope_dims(list(srcs) + list(dsts))
    T = srcs[0].shape[0]
    if any(s.shape[0] != T for s in srcs) or any(t.shape[0] < int(n) for t in dsts) or idx.numel() < int(n):
        raise ValueError("srcs share T rows; dsts hold n rows; idx n entries")
    st = lib().ut_fg_gather_rope(_p(idx), int(n), len(srcs), _ptr_array(srcs), _ptr_array(dsts), T, H, d, dtype,
                                 ctypes.byref(rope), _stream())
    _check("ut_fg_gather_rope", st)
    return dsts


def ut_fg_scatter_rope(idx: torch.Tensor, n: int, srcs: Sequence[torch.Tensor], dsts: Sequence[torch.Tensor],
                       rope: Rope, bg_mode: int = UT_BG_ZERO) -> None:
    """Inverse-rotated scatter: dst[idx[i]] = R(idx[i])^T src[i]; background rows per bg_mode (KEEP / ZERO)."""
    H, d, dtype = _rope_dims(list(srcs) + list(dsts))
    T = dsts[0].shape[0]
    if any(t.shape[0] != T for t in dsts) or any(s.shape[0] < int(n) for s in srcs) or idx.numel() < int(n):
        raise ValueError("dsts share T rows; srcs hold n rows; idx n entries")
    st = lib().ut_fg_scatter_rope(_p(idx), int(n), len(srcs), _ptr_array(srcs), _ptr_array(dsts), T, H, d, dtype,
                                  ctypes.byref(rope), bg_mode, _stream())
    _check("ut_fg_scatter_rope", st)


def ut_fg_euler_update(idx: torch.Tensor, n: int, z: torch.Tensor, v: torch.Tensor, dt: float,
                       status: Optional[torch.Tensor] = None) -> None:
    """Sparse Euler step in place: z[idx[i]] += dt * v[i] for i < n (dt = t_prev - t_curr)."""
    if z.dtype not in (torch.bfloat16, torch.float32) or v.dtype != z.dtype:
        raise ValueError("z and v must share dtype bf16 or fp32")
    if not (z.is_contiguous() and v.is_contiguous()):
        raise ValueError("z and v must be contiguous")
    T = z.shape[0]
    C = z[0].numel() if T > 0 else (v[0].numel() if v.shape[0] > 0 else 0)
    if (v.shape[0] > 0 and v[0].numel() != C) or v.shape[0] < int(n) or idx.numel() < int(n):
        raise ValueError("v must hold n rows of z's row size; idx n entries")
    dtype = UT_BF16 if z.dtype == torch.bfloat16 else UT_F32
    st = lib().ut_fg_euler_update(_p(idx), int(n), _p(z), _p(v), T, C, dtype, float(dt), _p(status), _stream())
    _check("ut_fg_euler_update", st)


def ut_fg_euler_update_gather(idx: torch.Tensor, n: int, z: torch.Tensor, v: torch.Tensor, dt: float,
                              zc: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Sparse Euler step in place and the gather of the updated rows:
    z[idx[i]] += dt * v[i]; zc[i] = z[idx[i]] for i < n.  Returns zc."""
    if z.dtype not in (torch.bfloat16, torch.float32) or v.dtype != z.dtype:
        raise ValueError("z and v must share dtype bf16 or fp32")
    if not (z.is_contiguous() and v.is_contiguous()):
        raise ValueError("z and v must be contiguous")
    T = z.shape[0]
    C = z[0].numel() if T > 0 else (v[0].numel() if v.shape[0] > 0 else 0)
    if (v.shape[0] > 0 and v[0].numel() != C) or v.shape[0] < int(n) or idx.numel() < int(n):
        raise ValueError("v must hold n rows of z's row size; idx n entries")
    if zc is None:
        zc = torch.empty((max(int(n), 1),) + tuple(z.shape[1:]), dtype=z.dtype, device=z.device)
    if not zc.is_contiguous() or zc.dtype != z.dtype or zc.shape[0] < int(n) or (zc.shape[0] and zc[0].numel() != C):
        raise ValueError("zc must be contiguous with n rows of z's row size and dtype")
    dtype = UT_BF16 if z.dtype == torch.bfloat16 else UT_F32
    st = lib().ut_fg_euler_update_gather(_p(idx), int(n), _p(z), _p(v), _p(zc), T, C, dtype, float(dt), _p(status),
                                         _stream())
    _check("ut_fg_euler_update_gather", st)
    return zc


def ut_fg_composite(mask: torch.Tensor, z: torch.Tensor, z_bg: torch.Tensor) -> None:
    """Composite latent in place: background row t of z becomes z_bg[t % len(z_bg)]."""
    if not (z.is_contiguous() and z_bg.is_contiguous()):
        raise ValueError("z and z_bg must be contiguous")
    T = z.shape[0]
    row_bytes = z[0].numel() * z.element_size() if T > 0 else 0
    P = z_bg.shape[0]
    if P < 1 or z_bg[0].numel() * z_bg.element_size() != row_bytes or mask.numel() < T:
        raise ValueError("z_bg must hold rows of z's row size; mask T entries")
    st = lib().ut_fg_composite(_p(mask), T, _p(z), _p(z_bg), P, row_bytes, _stream())
    _check("ut_fg_composite", st)


def ut_block_mask(shape: AttnShape, mode: int, q: Optional[torch.Tensor] = None, k: Optional[torch.Tensor] = None,
                  rho: float = 0.0, bitmap: Optional[torch.Tensor] = None, col_cap: Optional[int] = None,
                  with_transpose: bool = True, status: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                  out: Optional[tuple] = None):
    """Key-block lists.  Returns (row_ptr, col_idx, col_ptr_t, row_idx_t) (the last two None if not asked)."""
    nq = -(-shape.n_tokens // shape.block)
    nk = -(-shape.n_tokens // (shape.block_k or shape.block))
    H = shape.n_heads
    dev = (q if q is not None else bitmap).device
    L = lib()
    if col_cap is None:
        col_cap = H * nq * (ut_topk_count(rho, nk) if mode == UT_MASK_TOPK else nk)
    if out is None:
        row_ptr = torch.empty(H * nq + 1, dtype=torch.int32, device=dev)
        col_idx = torch.empty(max(col_cap, 1), dtype=torch.int32, device=dev)
        col_ptr = torch.empty(H * nk + 1, dtype=torch.int32, device=dev) if with_transpose else None
        row_idx = torch.empty(max(col_cap, 1), dtype=torch.int32, device=dev) if with_transpose else None
    else:
        row_ptr, col_idx, col_ptr, row_idx = out
    wsb = L.ut_block_mask_workspace_size(ctypes.byref(shape), mode)
    if ws is None:
        ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device=dev)
    if status is None and mode == UT_MASK_BITMAP:
        status = status_word(dev)
    st = L.ut_block_mask(ctypes.byref(shape), mode, _p(q), _p(k), float(rho), _p(bitmap), _p(row_ptr), _p(col_idx),
                         col_cap, _p(col_ptr), _p(row_idx), _p(ws), ws.numel(), _p(status), _stream())
    _check("ut_block_mask", st)
    return row_ptr, col_idx, col_ptr, row_idx


def ut_bsattn_fwd(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, row_ptr: torch.Tensor, col_idx: torch.Tensor,
                  block: int, softmax_scale: Optional[float] = None, o: Optional[torch.Tensor] = None,
                  lse: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None, block_k: int = 0):
    """Block-sparse attention forward (query blocks of `block` rows, key blocks of
    `block_k` rows, 0: same).  Returns (O [N,H,d], LSE [H,N] fp32)."""
    shape = attn_shape(q, block, block_k)
    N, H, d = q.shape
    scale = d ** -0.5 if softmax_scale is None else float(softmax_scale)
    if o is None:
        o = torch.empty_like(q)
    if lse is None:
        lse = torch.empty((H, N), dtype=torch.float32, device=q.device)
    st = lib().ut_bsattn_fwd(ctypes.byref(shape), _p(q), _p(k), _p(v), _p(row_ptr), _p(col_idx), scale, _p(o),
                             _p(lse), _p(status), _stream())
    _check("ut_bsattn_fwd", st)
    return o, lse


def ut_bsattn_bwd(q, k, v, o, lse, dout, row_ptr, col_idx, col_ptr_t, row_idx_t, block: int,
                  softmax_scale: Optional[float] = None, dq=None, dk=None, dv=None, ws=None, status=None,
                  block_k: int = 0):
    """Gradient of ut_bsattn_fwd.  Returns (dQ, dK, dV)."""
    shape = attn_shape(q, block, block_k)
    d = q.shape[2]
    scale = d ** -0.5 if softmax_scale is None else float(softmax_scale)
    dq = torch.empty_like(q) if dq is None else dq
    dk = torch.empty_like(k) if dk is None else dk
    dv = torch.empty_like(v) if dv is None else dv
    L = lib()
    wsb = L.ut_bsattn_bwd_workspace_size(ctypes.byref(shape))
    if ws is None:
        ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device=q.device)
    st = L.ut_bsattn_bwd(ctypes.byref(shape), _p(q), _p(k), _p(v), _p(o), _p(lse), _p(dout), _p(row_ptr),
                         _p(col_idx), _p(col_ptr_t), _p(row_idx_t), scale, _p(dq), _p(dk), _p(dv), _p(ws),
                         ws.numel(), _p(status), _stream())
    _check("ut_bsattn_bwd", st)
    return dq, dk, dv

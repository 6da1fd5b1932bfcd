"""Python binding of libqmla, the GB300 (sm_103a) low-bit MLA decode library.

Argument marshalling only: every step of the path runs in the library's CUDA
kernels; PyTorch supplies device memory and streams. The functions mirror the
C ABI of ``include/qmla.h`` (names without the ``qmla_`` prefix) and take
torch tensors. The library is loaded from ``lib/libqmla.so`` inside this
package (built by ``paper_2609_36760_gb300.build``); if it is missing every
call raises instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "lib", "libqmla.so")
_lib = None

OK = 0
STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported device or shape", 3: "workspace too small", 4: "CUDA error"}
DEVERR_BAD_BLOCK = 1
DEVERR_BAD_POSITION = 2
DEVERR_BAD_SEQ = 4
DEVERR_TIMEOUT = 8


CACHE_KINDS = {4: 4, 2: 2, "c4r4": 5, "bf16": 16}  # qmla_decode_desc.cache_kind codes


class DecodeDesc(ctypes.Structure):
    """qmla_decode_desc (include/qmla.h), field for field."""
    _fields_ = [("pool", ctypes.c_void_p), ("cache_kind", ctypes.c_int), ("num_blocks", ctypes.c_int),
                ("q_latent", ctypes.c_void_p), ("q_pe", ctypes.c_void_p), ("batch", ctypes.c_int),
                ("q_tokens", ctypes.c_int), ("heads", ctypes.c_int), ("block_table", ctypes.c_void_p),
                ("max_blocks", ctypes.c_int), ("seq_lens", ctypes.c_void_p), ("prot", ctypes.c_void_p),
                ("softmax_scale", ctypes.c_float), ("out", ctypes.c_void_p), ("lse", ctypes.c_void_p),
                ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t), ("dev_err", ctypes.c_void_p),
                ("ev_before_main", ctypes.c_void_p), ("ev_after_main", ctypes.c_void_p)]


class QmlaError(RuntimeError):
    def __init__(self, fn: str, status: int):
        extra = ""
        if status == 4 and _lib is not None:
            extra = f" (cudaError {_lib.qmla_last_cuda_error()})"
        super().__init__(f"{fn} failed: {STATUS.get(status, status)}{extra}")
        self.status = status


def library_path() -> str:
    return _LIB_PATH


def lib():
    """Loads libqmla.so (once). Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise RuntimeError(f"libqmla.so not found at {_LIB_PATH}; build it with "
                           "`python -m paper_2609_36760_gb300.build`")
    L = ctypes.CDLL(_LIB_PATH)
    vp, i32, sz, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_float
    L.qmla_block_bytes.argtypes, L.qmla_block_bytes.restype = [i32], sz
    L.qmla_bf16_block_bytes.argtypes, L.qmla_bf16_block_bytes.restype = [], sz
    L.qmla_quant_append.argtypes = [vp, i32, i32, vp, vp, vp, vp, i32, vp, i32, i32, vp, vp]
    L.qmla_quant_append.restype = i32
    L.qmla_bf16_append.argtypes = [vp, i32, vp, vp, vp, vp, i32, vp, i32, i32, vp, vp]
    L.qmla_bf16_append.restype = i32
    L.qmla_decode_workspace_bytes.argtypes, L.qmla_decode_workspace_bytes.restype = [i32, i32], sz
    L.qmla_mla_decode.argtypes = [vp, i32, i32, vp, vp, i32, i32, vp, i32, vp, f32, vp, vp, vp, sz, vp, vp]
    L.qmla_mla_decode.restype = i32
    L.qmla_mla_decode_bf16cache.argtypes = [vp, i32, vp, vp, i32, i32, vp, i32, vp, f32, vp, vp, vp, sz, vp, vp]
    L.qmla_mla_decode_bf16cache.restype = i32
    L.qmla_read_dev_err.argtypes, L.qmla_read_dev_err.restype = [vp, ctypes.POINTER(ctypes.c_uint32), vp], i32
    L.qmla_last_cuda_error.argtypes, L.qmla_last_cuda_error.restype = [], i32
    L.qmla_status_string.argtypes, L.qmla_status_string.restype = [i32], ctypes.c_char_p
    L.qmla_num_sms.argtypes, L.qmla_num_sms.restype = [], i32
    L.qmla_mla_decode_ex.argtypes, L.qmla_mla_decode_ex.restype = [ctypes.POINTER(DecodeDesc), vp], i32
    L.qmla_static_scratch_bytes.argtypes, L.qmla_static_scratch_bytes.restype = [], sz
    L.qmla_mla_decode_static.argtypes = [vp, i32, i32, vp, vp, i32, i32, vp, i32, vp, f32, vp, vp, vp, vp]
    L.qmla_mla_decode_static.restype = i32
    L.qmla_protect_bytes_per_seq.argtypes, L.qmla_protect_bytes_per_seq.restype = [], sz
    L.qmla_quant_append_protected.argtypes = [vp, i32, i32, vp, vp, vp, vp, i32, vp, i32, i32, vp, vp, vp, vp]
    L.qmla_quant_append_protected.restype = i32
    L.qmla_mla_decode_protected.argtypes = [vp, i32, i32, vp, vp, i32, i32, vp, i32, vp, vp, f32, vp, vp, vp, sz,
                                            vp, vp]
    L.qmla_mla_decode_protected.restype = i32
    L.qmla_mla_decode_multi.argtypes = [vp, i32, i32, vp, vp, i32, i32, i32, vp, i32, vp, vp, f32, vp, vp, vp, sz,
                                        vp, vp]
    L.qmla_mla_decode_multi.restype = i32
    L.qmla_debug_wait_timeout.argtypes = [ctypes.c_uint32, vp, vp]
    L.qmla_debug_wait_timeout.restype = i32
    L.qmla_debug_tile.argtypes = [vp, i32, i32, vp, i32, vp, i32, i32, i32, vp, vp, vp, vp]
    L.qmla_debug_tile.restype = i32
    L.qmla_c4r4_page_bytes.argtypes, L.qmla_c4r4_page_bytes.restype = [], sz
    L.qmla_quant_append_c4r4.argtypes = [vp, i32, vp, vp, vp, vp, i32, vp, i32, i32, vp, vp, vp, vp]
    L.qmla_quant_append_c4r4.restype = i32
    L.qmla_mla_decode_c4r4.argtypes = [vp, i32, vp, vp, i32, i32, vp, i32, vp, vp, f32, vp, vp, vp, sz, vp, vp]
    L.qmla_mla_decode_c4r4.restype = i32
    _lib = L
    return L


def _ptr(t: torch.Tensor | None):
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(fn: str, st: int) -> None:
    if st != OK:
        raise QmlaError(fn, st)


def block_bytes(c_bits: int) -> int:
    return int(lib().qmla_block_bytes(c_bits))


def bf16_block_bytes() -> int:
    return int(lib().qmla_bf16_block_bytes())


def num_sms() -> int:
    return int(lib().qmla_num_sms())


def decode_workspace_bytes(batch: int, heads: int) -> int:
    return int(lib().qmla_decode_workspace_bytes(batch, heads))


def quant_append(pool: torch.Tensor, c_bits: int, latent: torch.Tensor, k_pe: torch.Tensor,
                 seq_ids: torch.Tensor | None, positions: torch.Tensor, block_table: torch.Tensor,
                 dev_err: torch.Tensor, stream=None) -> None:
    """qmla_quant_append: pool uint8 [num_blocks, block_bytes]; latent bf16 [n,512];
    k_pe bf16 [n,64]; seq_ids/positions int32 [n]; block_table int32 [S, max_blocks]."""
    n = latent.shape[0]
    st = lib().qmla_quant_append(_ptr(pool), c_bits, pool.shape[0], _ptr(latent), _ptr(k_pe), _ptr(seq_ids),
                                 _ptr(positions), n, _ptr(block_table), block_table.shape[0],
                                 block_table.shape[1], _ptr(dev_err), _stream(stream))
    _check("qmla_quant_append", st)


def protect_bytes_per_seq() -> int:
    return int(lib().qmla_protect_bytes_per_seq())


def quant_append_protected(pool: torch.Tensor, c_bits: int, latent: torch.Tensor, k_pe: torch.Tensor,
                           seq_ids: torch.Tensor | None, positions: torch.Tensor, block_table: torch.Tensor,
                           seq_lens: torch.Tensor, prot: torch.Tensor, dev_err: torch.Tensor, stream=None) -> None:
    """qmla_quant_append_protected: quant_append plus the sink/recent bf16 rows;
    seq_lens int32 [S] = lengths after this call; prot [S, 132, 576] bf16."""
    n = latent.shape[0]
    st = lib().qmla_quant_append_protected(_ptr(pool), c_bits, pool.shape[0], _ptr(latent), _ptr(k_pe),
                                           _ptr(seq_ids), _ptr(positions), n, _ptr(block_table),
                                           block_table.shape[0], block_table.shape[1], _ptr(seq_lens), _ptr(prot),
                                           _ptr(dev_err), _stream(stream))
    _check("qmla_quant_append_protected", st)


def bf16_append(pool: torch.Tensor, latent: torch.Tensor, k_pe: torch.Tensor, seq_ids: torch.Tensor | None,
                positions: torch.Tensor, block_table: torch.Tensor, dev_err: torch.Tensor, stream=None) -> None:
    n = latent.shape[0]
    st = lib().qmla_bf16_append(_ptr(pool), pool.shape[0], _ptr(latent), _ptr(k_pe), _ptr(seq_ids),
                                _ptr(positions), n, _ptr(block_table), block_table.shape[0], block_table.shape[1],
                                _ptr(dev_err), _stream(stream))
    _check("qmla_bf16_append", st)


def mla_decode(pool: torch.Tensor, c_bits: int, q_latent: torch.Tensor, q_pe: torch.Tensor,
               block_table: torch.Tensor, seq_lens: torch.Tensor, softmax_scale: float, out: torch.Tensor,
               lse: torch.Tensor | None, workspace: torch.Tensor, dev_err: torch.Tensor, stream=None) -> None:
    """qmla_mla_decode: q_latent bf16 [B,H,512], q_pe bf16 [B,H,64], out f32 [B,H,512], lse f32 [B,H]."""
    B, H = q_latent.shape[0], q_latent.shape[1]
    st = lib().qmla_mla_decode(_ptr(pool), c_bits, pool.shape[0], _ptr(q_latent), _ptr(q_pe), B, H,
                               _ptr(block_table), block_table.shape[1], _ptr(seq_lens), float(softmax_scale),
                               _ptr(out), _ptr(lse), _ptr(workspace), workspace.numel() * workspace.element_size(),
                               _ptr(dev_err), _stream(stream))
    _check("qmla_mla_decode", st)


def mla_decode_protected(pool: torch.Tensor, c_bits: int, q_latent: torch.Tensor, q_pe: torch.Tensor,
                         block_table: torch.Tensor, seq_lens: torch.Tensor, prot: torch.Tensor, softmax_scale: float,
                         out: torch.Tensor, lse: torch.Tensor | None, workspace: torch.Tensor, dev_err: torch.Tensor,
                         stream=None) -> None:
    """qmla_mla_decode_protected: mla_decode with sink4/local128 bf16 rows from prot [B, 132, 576]."""
    B, H = q_latent.shape[0], q_latent.shape[1]
    st = lib().qmla_mla_decode_protected(_ptr(pool), c_bits, pool.shape[0], _ptr(q_latent), _ptr(q_pe), B, H,
                                         _ptr(block_table), block_table.shape[1], _ptr(seq_lens), _ptr(prot),
                                         float(softmax_scale), _ptr(out), _ptr(lse), _ptr(workspace),
                                         workspace.numel() * workspace.element_size(), _ptr(dev_err),
                                         _stream(stream))
    _check("qmla_mla_decode_protected", st)


def mla_decode_multi(pool: torch.Tensor, c_bits: int, q_latent: torch.Tensor, q_pe: torch.Tensor,
                     block_table: torch.Tensor, seq_lens: torch.Tensor, softmax_scale: float, out: torch.Tensor,
                     lse: torch.Tensor | None, workspace: torch.Tensor, dev_err: torch.Tensor,
                     prot: torch.Tensor | None = None, stream=None) -> None:
    """qmla_mla_decode_multi: q_latent bf16 [B,T,H,512], q_pe bf16 [B,T,H,64],
    out f32 [B,T,H,512], lse f32 [B,T,H]; workspace for B x (T*H) heads."""
    B, T, H = q_latent.shape[0], q_latent.shape[1], q_latent.shape[2]
    st = lib().qmla_mla_decode_multi(_ptr(pool), c_bits, pool.shape[0], _ptr(q_latent), _ptr(q_pe), B, T, H,
                                     _ptr(block_table), block_table.shape[1], _ptr(seq_lens), _ptr(prot),
                                     float(softmax_scale), _ptr(out), _ptr(lse), _ptr(workspace),
                                     workspace.numel() * workspace.element_size(), _ptr(dev_err), _stream(stream))
    _check("qmla_mla_decode_multi", st)


CACHE_C4R4 = 5   # qmla_debug_tile cache kinds (besides content bit widths 4 and 2)
CACHE_BF16 = 16


def debug_tile(pool: torch.Tensor, cache_kind: int, block_table: torch.Tensor, seq_lens: torch.Tensor, b: int,
               j: int, tile: torch.Tensor, dev_err: torch.Tensor, prot: torch.Tensor | None = None,
               stream=None) -> None:
    """qmla_debug_tile: tile j of sequence b as the decode kernel builds it, into
    tile [128, 576] (fp16 or int16)."""
    st = lib().qmla_debug_tile(_ptr(pool), cache_kind, pool.shape[0], _ptr(block_table), block_table.shape[1],
                               _ptr(seq_lens), block_table.shape[0], b, j, _ptr(prot), _ptr(tile), _ptr(dev_err),
                               _stream(stream))
    _check("qmla_debug_tile", st)


DEVERR_SITE_SOFTMAX = 0x100 << 5


def debug_wait_timeout(limit_us: int, dev_err: torch.Tensor, stream=None) -> None:
    """qmla_debug_wait_timeout: a decode wait that runs out after limit_us."""
    _check("qmla_debug_wait_timeout", lib().qmla_debug_wait_timeout(limit_us, _ptr(dev_err), _stream(stream)))


def c4r4_page_bytes() -> int:
    """Bytes of one 64-token page of the paper's INT4 format (20480)."""
    return int(lib().qmla_c4r4_page_bytes())


def quant_append_c4r4(pool: torch.Tensor, latent: torch.Tensor, k_pe: torch.Tensor, seq_ids: torch.Tensor | None,
                      positions: torch.Tensor, block_table: torch.Tensor, dev_err: torch.Tensor,
                      seq_lens: torch.Tensor | None = None, prot: torch.Tensor | None = None, stream=None) -> None:
    """qmla_quant_append_c4r4: pages of the paper's format; with prot (and
    seq_lens = lengths after this call) also the sink/recent bf16 rows."""
    n = latent.shape[0]
    st = lib().qmla_quant_append_c4r4(_ptr(pool), pool.shape[0], _ptr(latent), _ptr(k_pe), _ptr(seq_ids),
                                      _ptr(positions), n, _ptr(block_table), block_table.shape[0],
                                      block_table.shape[1], _ptr(seq_lens), _ptr(prot), _ptr(dev_err),
                                      _stream(stream))
    _check("qmla_quant_append_c4r4", st)


def mla_decode_c4r4(pool: torch.Tensor, q_latent: torch.Tensor, q_pe: torch.Tensor, block_table: torch.Tensor,
                    seq_lens: torch.Tensor, softmax_scale: float, out: torch.Tensor, lse: torch.Tensor | None,
                    workspace: torch.Tensor, dev_err: torch.Tensor, prot: torch.Tensor | None = None,
                    stream=None) -> None:
    """qmla_mla_decode_c4r4: mla_decode over pages of the paper's format, with
    sink4/local128 protection when prot [B, 132, 576] is given."""
    B, H = q_latent.shape[0], q_latent.shape[1]
    st = lib().qmla_mla_decode_c4r4(_ptr(pool), pool.shape[0], _ptr(q_latent), _ptr(q_pe), B, H, _ptr(block_table),
                                    block_table.shape[1], _ptr(seq_lens), _ptr(prot), float(softmax_scale),
                                    _ptr(out), _ptr(lse), _ptr(workspace),
                                    workspace.numel() * workspace.element_size(), _ptr(dev_err), _stream(stream))
    _check("qmla_mla_decode_c4r4", st)


def mla_decode_bf16cache(pool: torch.Tensor, q_latent: torch.Tensor, q_pe: torch.Tensor, block_table: torch.Tensor,
                         seq_lens: torch.Tensor, softmax_scale: float, out: torch.Tensor, lse: torch.Tensor | None,
                         workspace: torch.Tensor, dev_err: torch.Tensor, stream=None) -> None:
    B, H = q_latent.shape[0], q_latent.shape[1]
    st = lib().qmla_mla_decode_bf16cache(_ptr(pool), pool.shape[0], _ptr(q_latent), _ptr(q_pe), B, H,
                                         _ptr(block_table), block_table.shape[1], _ptr(seq_lens),
                                         float(softmax_scale), _ptr(out), _ptr(lse), _ptr(workspace),
                                         workspace.numel() * workspace.element_size(), _ptr(dev_err),
                                         _stream(stream))
    _check("qmla_mla_decode_bf16cache", st)


def mla_decode_static(pool: torch.Tensor, c_bits: int, q_latent: torch.Tensor, q_pe: torch.Tensor,
                      block_table: torch.Tensor, seq_lens: torch.Tensor, softmax_scale: float, out: torch.Tensor,
                      lse: torch.Tensor | None, dev_err: torch.Tensor, stream=None) -> None:
    """qmla_mla_decode_static: qmla_mla_decode for callers that cannot allocate a
    workspace; uses the library's fixed device scratch (see include/qmla.h)."""
    B, H = q_latent.shape[0], q_latent.shape[1]
    st = lib().qmla_mla_decode_static(_ptr(pool), c_bits, pool.shape[0], _ptr(q_latent), _ptr(q_pe), B, H,
                                      _ptr(block_table), block_table.shape[1], _ptr(seq_lens),
                                      float(softmax_scale), _ptr(out), _ptr(lse), _ptr(dev_err), _stream(stream))
    _check("qmla_mla_decode_static", st)


def static_scratch_bytes() -> int:
    return int(lib().qmla_static_scratch_bytes())


def mla_decode_ex(pool: torch.Tensor, cache_kind, q_latent: torch.Tensor, q_pe: torch.Tensor,
                  block_table: torch.Tensor, seq_lens: torch.Tensor, softmax_scale: float, out: torch.Tensor,
                  lse: torch.Tensor | None, workspace: torch.Tensor, dev_err: torch.Tensor, prot=None,
                  events: tuple | None = None, stream=None) -> None:
    """qmla_mla_decode_ex: cache_kind 4, 2, "c4r4" or "bf16"; q_latent [B,H,512] or
    [B,T,H,512]; events = (before_main, after_main) torch.cuda.Event pair (already
    recorded once, so that they exist) to record around this call's main kernel."""
    if q_latent.dim() == 3:
        B, T, H = q_latent.shape[0], 1, q_latent.shape[1]
    else:
        B, T, H = q_latent.shape[0], q_latent.shape[1], q_latent.shape[2]
    d = DecodeDesc()
    d.pool, d.cache_kind, d.num_blocks = _ptr(pool), CACHE_KINDS[cache_kind], pool.shape[0]
    d.q_latent, d.q_pe, d.batch, d.q_tokens, d.heads = _ptr(q_latent), _ptr(q_pe), B, T, H
    d.block_table, d.max_blocks, d.seq_lens = _ptr(block_table), block_table.shape[1], _ptr(seq_lens)
    d.prot, d.softmax_scale, d.out, d.lse = _ptr(prot), float(softmax_scale), _ptr(out), _ptr(lse)
    d.workspace, d.workspace_bytes = _ptr(workspace), workspace.numel() * workspace.element_size()
    d.dev_err = _ptr(dev_err)
    if events is not None:
        d.ev_before_main = ctypes.c_void_p(events[0].cuda_event) if events[0] is not None else None
        d.ev_after_main = ctypes.c_void_p(events[1].cuda_event) if events[1] is not None else None
    _check("qmla_mla_decode_ex", lib().qmla_mla_decode_ex(ctypes.byref(d), _stream(stream)))


def read_dev_err(dev_err: torch.Tensor, stream=None) -> int:
    out = ctypes.c_uint32(0)
    _check("qmla_read_dev_err", lib().qmla_read_dev_err(_ptr(dev_err), ctypes.byref(out), _stream(stream)))
    return int(out.value)


def workspace_for(batch: int, heads: int, device="cuda") -> torch.Tensor:
    """A workspace tensor of the size qmla_mla_decode needs (256-byte aligned)."""
    n = decode_workspace_bytes(batch, heads)
    if n == 0:
        raise QmlaError("qmla_decode_workspace_bytes", 2)
    return torch.empty(n, dtype=torch.uint8, device=device)

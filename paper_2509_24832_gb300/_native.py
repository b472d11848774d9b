"""ctypes binding of libsemshare.so (the C ABI declared in include/semshare.h).

Argument marshalling only: every step of the path runs in the library's CUDA kernels.
PyTorch supplies device memory and the current stream.  There is no fallback: if the
library is missing the call raises."""
from __future__ import annotations

import ctypes
import os
import threading
from typing import NamedTuple

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
# SEMSHARE_CHECKED=1 in the environment (read once, at import) selects the checked build, whose
# kernels also verify their pipeline bookkeeping (semshare_checked_build in include/semshare.h)
CHECKED = os.environ.get("SEMSHARE_CHECKED", "") not in ("", "0")
LIB_PATH = os.path.join(_PKG, "_lib", "libsemshare_checked.so" if CHECKED else "libsemshare.so")

OK, EINVAL, EUNSUPPORTED, ECUDA, EINDEX, ETIMEOUT, ETOOLARGE, ECHECK = range(8)
MATCH_STATIC_MAX_TARGETS = 262144
FLAG_INDEX, FLAG_TIMEOUT, FLAG_CHECK = 1, 2, 4
KERNEL_HASH_2SM, KERNEL_HASH, KERNEL_HAMMING_TC, KERNEL_SELFTEST = 1, 2, 3, 15
BF16, F32 = 0, 1
ROPE_LAYOUTS = {"interleaved": 0, "half": 1, "none": 2}

_lock = threading.Lock()
_lib = None


class SemshareError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


class KVLayout(ctypes.Structure):
    """semshare_kv_layout: element (b, l, h, t, e) at b*stride_batch + l*stride_layer +
    h*stride_head + t*stride_token + e (strides in elements)."""
    _fields_ = [("n_layers", ctypes.c_int32), ("n_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("elem_bytes", ctypes.c_int32), ("stride_batch", ctypes.c_int64), ("stride_layer", ctypes.c_int64),
                ("stride_head", ctypes.c_int64), ("stride_token", ctypes.c_int64)]


def load():
    """Loads libsemshare.so (built in-tree by paper_2509_24832_gb300.build)."""
    global _lib
    lib = _lib
    if lib is not None:  # the common case, without the lock
        return lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it first (python -c 'import __graft_entry__ as g; g.build()')")
        lib = ctypes.CDLL(LIB_PATH)
        P, i32, i64, u32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
        lib.semshare_status_string.argtypes = [ctypes.c_int]
        lib.semshare_status_string.restype = ctypes.c_char_p
        lib.semshare_flag_status.argtypes = [u32]
        lib.semshare_flag_status.restype = ctypes.c_int
        lib.semshare_abi_version.restype = i32
        lib.semshare_checked_build.restype = i32
        lib.semshare_check_selftest.argtypes = [P, P]
        lib.semshare_check_selftest.restype = ctypes.c_int
        lib.semshare_rope_table.argtypes = [i32, ctypes.c_double, P, P]
        lib.semshare_rope_table.restype = ctypes.c_int
        lib.semshare_hash_pair_workspace_size.argtypes = [i64, i32, i32]
        lib.semshare_hash_pair_workspace_size.restype = ctypes.c_size_t
        lib.semshare_hash_pair.argtypes = [P, ctypes.c_int, i64, i32, i64, P, P, P, i32, P, P, P, ctypes.c_size_t, P, P]
        lib.semshare_hash_pair.restype = ctypes.c_int
        lib.semshare_hash_workspace_size.argtypes = [i64, i32, i32]
        lib.semshare_hash_workspace_size.restype = ctypes.c_size_t
        lib.semshare_hash.argtypes = [P, ctypes.c_int, i64, i32, i64, P, P, P, i32, P, P, P, ctypes.c_size_t, P, P]
        lib.semshare_hash.restype = ctypes.c_int
        lib.semshare_hash_ex.argtypes = [P, ctypes.c_int, i64, i32, i64, P, P, P, i32, u32, P, P, P, ctypes.c_size_t,
                                         P, P]
        lib.semshare_hash_ex.restype = ctypes.c_int
        lib.semshare_signs_pitch.argtypes = [i32]
        lib.semshare_signs_pitch.restype = i32
        lib.semshare_hash_signs.argtypes = [P, ctypes.c_int, i64, i32, i64, P, P, P, i32, u32, P, P, P, P,
                                            ctypes.c_size_t, P, P]
        lib.semshare_hash_signs.restype = ctypes.c_int
        lib.semshare_match_tc_signs_workspace_size.argtypes = [i64]
        lib.semshare_match_tc_signs_workspace_size.restype = ctypes.c_size_t
        lib.semshare_match_tc_signs.argtypes = [P, i64, P, i64, i32, P, P, P, ctypes.c_size_t, P, P]
        lib.semshare_match_tc_signs.restype = ctypes.c_int
        lib.semshare_match_workspace_size.argtypes = [i64]
        lib.semshare_match_workspace_size.restype = ctypes.c_size_t
        lib.semshare_match.argtypes = [P, i64, P, i64, i32, P, P, P, ctypes.c_size_t, P]
        lib.semshare_match.restype = ctypes.c_int
        lib.semshare_match_tc_workspace_size.argtypes = [i64, i64, i32]
        lib.semshare_match_tc_workspace_size.restype = ctypes.c_size_t
        lib.semshare_match_tc.argtypes = [P, i64, P, i64, i32, P, P, P, ctypes.c_size_t, P, P]
        lib.semshare_match_tc.restype = ctypes.c_int
        lib.semshare_retrieve_workspace_size.argtypes = [i64, i64, i32, i32]
        lib.semshare_retrieve_workspace_size.restype = ctypes.c_size_t
        lib.semshare_retrieve.argtypes = [P, i64, P, P, i32, i32, ctypes.c_double, ctypes.c_double, P, P, P, P, P, P,
                                          P, ctypes.c_size_t, P, P]
        lib.semshare_retrieve.restype = ctypes.c_int
        lib.semshare_match_static.argtypes = [P, i64, P, i64, i32, P, P, P]
        lib.semshare_match_tc_selected_workspace_size.argtypes = [i64, P, i32, i32]
        lib.semshare_match_tc_selected_workspace_size.restype = ctypes.c_size_t
        lib.semshare_match_tc_selected.argtypes = [P, i64, P, P, i32, P, i32, P, P, P, ctypes.c_size_t, P, P]
        lib.semshare_match_tc_selected.restype = ctypes.c_int
        lib.semshare_match_static.restype = ctypes.c_int
        lib.semshare_gather_kv.argtypes = [P, P, P, i32, KVLayout, P, i64, i32, P, P, KVLayout, P, P]
        lib.semshare_gather_kv.restype = ctypes.c_int
        lib.semshare_gather_kv_retained.argtypes = [P, P, P, i32, KVLayout, P, i64, P, P, P, P, KVLayout, P, P]
        lib.semshare_gather_kv_retained.restype = ctypes.c_int
        lib.semshare_fetch_workspace_size.argtypes = [i64]
        lib.semshare_fetch_workspace_size.restype = ctypes.c_size_t
        lib.semshare_fetch_rows.argtypes = [P, P, P, P, P, i32, KVLayout, P, i64, P, ctypes.c_size_t, P, P]
        lib.semshare_fetch_rows.restype = ctypes.c_int
        lib.semshare_kv_deviation.argtypes = [P, P, KVLayout, P, P, KVLayout, ctypes.c_int, i64, P, P, P, P]
        lib.semshare_kv_deviation.restype = ctypes.c_int
        lib.semshare_select_hd.argtypes = [P, i32, i64, i64, P, P, P]
        lib.semshare_select_hd.restype = ctypes.c_int
        lib.semshare_hd_count.argtypes = [i64, i32]
        lib.semshare_hd_count.restype = i64
        lib.semshare_retain_counts.argtypes = [i64, P, i32, i32, P]
        lib.semshare_retain_counts.restype = ctypes.c_int
        _lib = lib
        return lib


def status_string(status: int) -> str:
    try:
        return load().semshare_status_string(int(status)).decode()
    except RuntimeError:
        return f"status {status}"


def _check(status: int, where: str):
    if status != OK:
        raise SemshareError(status, where)


def _ptr(t: torch.Tensor | None):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _current_raw_stream() -> int:
    """The current CUDA stream of the current device as a raw handle (what
    torch.cuda.current_stream().cuda_stream returns, without building a Stream object)."""
    return torch._C._cuda_getCurrentRawStream(torch._C._cuda_getDevice())


def _stream(stream) -> ctypes.c_void_p:
    return ctypes.c_void_p(_current_raw_stream() if stream is None else stream.cuda_stream)


class Prepared:
    """A library call whose arguments were checked and marshalled once (`prepare=True` on
    semshare_hash, semshare_match_tc, semshare_gather_kv).  Calling it enqueues the same work on
    the current stream (or `stream`) and returns the call's outputs, for a few microseconds of
    host time instead of the binding's checks.  It keeps its tensors alive; their storage must
    not be resized or reallocated while it is used."""

    __slots__ = ("_fn", "_args", "_where", "_keep", "result")

    def __init__(self, fn, args, where, keep, result):
        self._fn, self._args, self._where, self._keep, self.result = fn, args, where, keep, result

    def __call__(self, stream=None):
        st = self._fn(*self._args, _stream(stream))
        if st != OK:
            raise SemshareError(st, self._where)
        return self.result


def _need_cuda(t: torch.Tensor, name: str):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")


def _need_device_accessible(t: torch.Tensor, name: str):
    """A CUDA tensor, or a pinned (page-locked) host tensor: the GPU reads it in place over the
    host link (its address is valid on the device)."""
    if not isinstance(t, torch.Tensor) or not (t.is_cuda or t.is_pinned()):
        raise ValueError(f"{name} must be a CUDA tensor or a pinned host tensor")


def new_err_flag(device=None) -> torch.Tensor:
    """A zeroed device word for the kernels' error bits."""
    return torch.zeros(1, dtype=torch.int32, device=device or "cuda")


def flag_status(err_flag: torch.Tensor) -> int:
    """Reads an error word back (synchronising on it) and maps its bits to a status."""
    return int(load().semshare_flag_status(int(err_flag.item()) & 0xFFFFFFFF))


def check_flag(err_flag: torch.Tensor, where: str = "kernel"):
    _check(flag_status(err_flag), where)


def semshare_abi_version() -> int:
    return int(load().semshare_abi_version())


def semshare_checked_build() -> bool:
    """True when the loaded library is the checked build."""
    return bool(load().semshare_checked_build())


def semshare_check_selftest(err_flag: torch.Tensor, stream=None) -> None:
    """Checked build: enqueue a kernel whose check fails on purpose (see include/semshare.h)."""
    _need_cuda(err_flag, "err_flag")
    _check(load().semshare_check_selftest(_ptr(err_flag), _stream(stream)), "semshare_check_selftest")


def check_record(err_flag_value: int) -> tuple[int, int]:
    """(kernel id, source line) of the first failed check packed into an err_flag word."""
    v = int(err_flag_value) & 0xFFFFFFFF
    return (v >> 8) & 0xFF, v >> 16


def semshare_rope_table(d: int, rope_base: float = 10000.0, out: torch.Tensor | None = None, device=None,
                        stream=None) -> torch.Tensor:
    """Rotation table for semshare_hash: [d] uint64 words (int64 storage): d/2 fixed-point turn
    fractions, then d/2 (cos, sin) pairs of the 32-position rotation."""
    if out is None:
        out = torch.empty(d, dtype=torch.int64, device=device or "cuda")
    _need_cuda(out, "out")
    _check(load().semshare_rope_table(int(d), float(rope_base), _ptr(out), _stream(stream)), "semshare_rope_table")
    return out


_hash_ws = {}


def semshare_hash_workspace_size(n: int, d: int, nbits: int) -> int:
    return int(load().semshare_hash_workspace_size(int(n), int(d), int(nbits)))


def hash_workspace(n: int, d: int, nbits: int, device=None) -> torch.Tensor:
    """A zero-filled hash workspace large enough for (n, d, nbits), kept per device and grown on
    demand.  The library leaves it zero-filled after every successful call, so calls issued one
    after another (on one stream) can share it; concurrent calls need their own."""
    dev = torch.device(device or "cuda")
    if dev.index is None:
        dev = torch.device("cuda", torch.cuda.current_device())
    need = max(256, semshare_hash_workspace_size(n, d, nbits))
    ws = _hash_ws.get(dev)
    if ws is None or ws.numel() < need:
        ws = torch.zeros(need, dtype=torch.uint8, device=dev)
        _hash_ws[dev] = ws
    return ws


def semshare_hash(emb: torch.Tensor, rope_table: torch.Tensor, hyperplanes: torch.Tensor,
                  positions: torch.Tensor | None = None, codes: torch.Tensor | None = None,
                  proj_out: torch.Tensor | None = None, err_flag: torch.Tensor | None = None,
                  workspace: torch.Tensor | None = None, stream=None, rope_layout: str = "interleaved",
                  *, prepare: bool = False):
    """LSH codes of RoPE-encoded rows.  emb [n][d] bf16/fp32 (rows may be strided),
    hyperplanes [nbits][d] bf16, positions [n] int32 (None: 0..n-1).  workspace: a zero-filled
    uint8 device buffer (default: the per-device one of hash_workspace()).  rope_layout:
    "interleaved" (pairs (2k, 2k+1), Eq. 1), "half" (pairs (k, k + d/2); bf16 rows, d a
    multiple of 128) or "none" (no rotation: rope_table and positions are ignored and may be
    None).  Returns codes [n][nbits/32] int32 (uint32 bit patterns)."""
    _need_cuda(emb, "emb")
    _need_cuda(hyperplanes, "hyperplanes")
    if emb.dim() != 2 or emb.stride(1) != 1:
        raise ValueError("emb must be [n][d] with unit stride along d")
    if emb.dtype == torch.bfloat16:
        dt = BF16
    elif emb.dtype == torch.float32:
        dt = F32
    else:
        raise ValueError("emb must be bfloat16 or float32")
    if hyperplanes.dtype != torch.bfloat16 or not hyperplanes.is_contiguous():
        raise ValueError("hyperplanes must be contiguous bfloat16 [nbits][d]")
    n, d = emb.shape
    nbits = hyperplanes.shape[0]
    if hyperplanes.shape[1] != d:
        raise ValueError("hyperplanes width differs from emb")
    if positions is not None:
        if positions.dtype != torch.int32 or positions.numel() != n or not positions.is_contiguous():
            raise ValueError("positions must be contiguous int32 [n]")
    if codes is None:
        codes = torch.empty((n, nbits // 32), dtype=torch.int32, device=emb.device)
    if workspace is None:
        workspace = hash_workspace(n, d, nbits, emb.device)
    ws_bytes = workspace.numel() * workspace.element_size()
    if rope_layout not in ROPE_LAYOUTS:
        raise ValueError(f"rope_layout must be one of {sorted(ROPE_LAYOUTS)}")
    if rope_layout != "none":
        _need_cuda(rope_table, "rope_table")
    args = (_ptr(emb), dt, n, d, emb.stride(0), _ptr(positions), _ptr(rope_table), _ptr(hyperplanes), nbits,
            ROPE_LAYOUTS[rope_layout], _ptr(codes), _ptr(proj_out), _ptr(workspace), ws_bytes, _ptr(err_flag))
    call = Prepared(load().semshare_hash_ex, args, "semshare_hash",
                    (emb, positions, rope_table, hyperplanes, proj_out, workspace, err_flag), codes)
    return call if prepare else call(stream)


def semshare_signs_pitch(nbits: int) -> int:
    """Bytes per sign row of semshare_hash_signs (128 * ceil(nbits / 128))."""
    return int(load().semshare_signs_pitch(int(nbits)))


def semshare_hash_signs(emb: torch.Tensor, rope_table: torch.Tensor, hyperplanes: torch.Tensor,
                        positions: torch.Tensor | None = None, codes: torch.Tensor | None = None,
                        signs: torch.Tensor | None = None, proj_out: torch.Tensor | None = None,
                        err_flag: torch.Tensor | None = None, workspace: torch.Tensor | None = None, stream=None,
                        rope_layout: str = "interleaved", *, prepare: bool = False):
    """semshare_hash that also writes the codes as e4m3 +-1 rows, the operands of
    semshare_match_tc_signs.  Arguments as for semshare_hash, plus signs: uint8
    [n][semshare_signs_pitch(nbits)] (allocated when None).  Returns (codes, signs)."""
    _need_cuda(emb, "emb")
    _need_cuda(hyperplanes, "hyperplanes")
    if emb.dim() != 2 or emb.stride(1) != 1:
        raise ValueError("emb must be [n][d] with unit stride along d")
    dt = {torch.bfloat16: BF16, torch.float32: F32}.get(emb.dtype)
    if dt is None:
        raise ValueError("emb must be bfloat16 or float32")
    if hyperplanes.dtype != torch.bfloat16 or not hyperplanes.is_contiguous():
        raise ValueError("hyperplanes must be contiguous bfloat16 [nbits][d]")
    n, d = emb.shape
    nbits = hyperplanes.shape[0]
    if hyperplanes.shape[1] != d:
        raise ValueError("hyperplanes width differs from emb")
    if positions is not None and (positions.dtype != torch.int32 or positions.numel() != n
                                  or not positions.is_contiguous()):
        raise ValueError("positions must be contiguous int32 [n]")
    pitch = semshare_signs_pitch(nbits)
    if codes is None:
        codes = torch.empty((n, nbits // 32), dtype=torch.int32, device=emb.device)
    if signs is None:
        signs = torch.empty((n, pitch), dtype=torch.uint8, device=emb.device)
    elif signs.dtype != torch.uint8 or signs.shape != (n, pitch) or not signs.is_contiguous():
        raise ValueError(f"signs must be contiguous uint8 [{n}][{pitch}]")
    if workspace is None:
        workspace = hash_workspace(n, d, nbits, emb.device)
    if rope_layout not in ROPE_LAYOUTS:
        raise ValueError(f"rope_layout must be one of {sorted(ROPE_LAYOUTS)}")
    if rope_layout != "none":
        _need_cuda(rope_table, "rope_table")
    args = (_ptr(emb), dt, n, d, emb.stride(0), _ptr(positions), _ptr(rope_table), _ptr(hyperplanes), nbits,
            ROPE_LAYOUTS[rope_layout], _ptr(codes), _ptr(signs), _ptr(proj_out), _ptr(workspace),
            workspace.numel() * workspace.element_size(), _ptr(err_flag))
    call = Prepared(load().semshare_hash_signs, args, "semshare_hash_signs",
                    (emb, positions, rope_table, hyperplanes, proj_out, workspace, err_flag), (codes, signs))
    return call if prepare else call(stream)


def semshare_hash_pair_workspace_size(n: int, d: int, nbits: int) -> int:
    return int(load().semshare_hash_pair_workspace_size(int(n), int(d), int(nbits)))


def semshare_hash_pair(emb: torch.Tensor, rope_table: torch.Tensor, hyperplanes: torch.Tensor,
                       positions: torch.Tensor | None = None, codes_plain: torch.Tensor | None = None,
                       codes_rotary: torch.Tensor | None = None, err_flag: torch.Tensor | None = None,
                       workspace: torch.Tensor | None = None, stream=None):
    """The codes of the rows as they are and after RoPE (interleaved pairs), in one launch.
    Arguments as for semshare_hash.  Returns (codes_plain, codes_rotary), each [n][nbits/32] int32."""
    _need_cuda(emb, "emb")
    _need_cuda(hyperplanes, "hyperplanes")
    _need_cuda(rope_table, "rope_table")
    if emb.dim() != 2 or emb.stride(1) != 1:
        raise ValueError("emb must be [n][d] with unit stride along d")
    dt = {torch.bfloat16: BF16, torch.float32: F32}.get(emb.dtype)
    if dt is None:
        raise ValueError("emb must be bfloat16 or float32")
    if hyperplanes.dtype != torch.bfloat16 or not hyperplanes.is_contiguous():
        raise ValueError("hyperplanes must be contiguous bfloat16 [nbits][d]")
    n, d = emb.shape
    nbits = hyperplanes.shape[0]
    if hyperplanes.shape[1] != d:
        raise ValueError("hyperplanes width differs from emb")
    if positions is not None and (positions.dtype != torch.int32 or positions.numel() != n
                                  or not positions.is_contiguous()):
        raise ValueError("positions must be contiguous int32 [n]")
    if codes_plain is None:
        codes_plain = torch.empty((n, nbits // 32), dtype=torch.int32, device=emb.device)
    if codes_rotary is None:
        codes_rotary = torch.empty((n, nbits // 32), dtype=torch.int32, device=emb.device)
    if workspace is None:
        workspace = hash_workspace(2 * ((n + 127) // 128) * 128, d, nbits, emb.device)
    st = load().semshare_hash_pair(_ptr(emb), dt, n, d, emb.stride(0), _ptr(positions), _ptr(rope_table),
                                   _ptr(hyperplanes), nbits, _ptr(codes_plain), _ptr(codes_rotary), _ptr(workspace),
                                   workspace.numel() * workspace.element_size(), _ptr(err_flag), _stream(stream))
    _check(st, "semshare_hash_pair")
    return codes_plain, codes_rotary


def semshare_match_workspace_size(n_tgt: int) -> int:
    return int(load().semshare_match_workspace_size(int(n_tgt)))


def semshare_match(tgt_codes: torch.Tensor, ref_codes: torch.Tensor, idx: torch.Tensor | None = None,
                   dist: torch.Tensor | None = None, workspace: torch.Tensor | None = None, nbits: int | None = None,
                   stream=None):
    """Hamming nearest reference row per target row (ties to the lowest index).
    Returns (idx int32 [n_tgt], dist int32 [n_tgt])."""
    _need_cuda(tgt_codes, "tgt_codes")
    _need_cuda(ref_codes, "ref_codes")
    if not tgt_codes.is_contiguous() or not ref_codes.is_contiguous():
        raise ValueError("codes must be contiguous")
    n_tgt, w = tgt_codes.shape
    n_ref = ref_codes.shape[0]
    if ref_codes.shape[1] != w:
        raise ValueError("code widths differ")
    nbits = 32 * w if nbits is None else nbits
    dev = tgt_codes.device
    if idx is None:
        idx = torch.empty(n_tgt, dtype=torch.int32, device=dev)
    if dist is None:
        dist = torch.empty(n_tgt, dtype=torch.int32, device=dev)
    ws_bytes = semshare_match_workspace_size(n_tgt)
    if workspace is None:
        workspace = torch.empty(max(ws_bytes, 8), dtype=torch.uint8, device=dev)
    st = load().semshare_match(_ptr(tgt_codes), n_tgt, _ptr(ref_codes), n_ref, nbits, _ptr(idx), _ptr(dist),
                               _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream))
    _check(st, "semshare_match")
    return idx, dist


def semshare_match_tc_workspace_size(n_tgt: int, n_ref: int, nbits: int) -> int:
    return int(load().semshare_match_tc_workspace_size(int(n_tgt), int(n_ref), int(nbits)))


def semshare_match_tc(tgt_codes: torch.Tensor, ref_codes: torch.Tensor, idx: torch.Tensor | None = None,
                      dist: torch.Tensor | None = None, workspace: torch.Tensor | None = None,
                      err_flag: torch.Tensor | None = None, nbits: int | None = None, stream=None, *,
                      prepare: bool = False):
    """semshare_match computed on the tensor cores (same result).  Returns (idx, dist)."""
    _need_cuda(tgt_codes, "tgt_codes")
    _need_cuda(ref_codes, "ref_codes")
    if not tgt_codes.is_contiguous() or not ref_codes.is_contiguous():
        raise ValueError("codes must be contiguous")
    n_tgt, w = tgt_codes.shape
    n_ref = ref_codes.shape[0]
    if ref_codes.shape[1] != w:
        raise ValueError("code widths differ")
    nbits = 32 * w if nbits is None else nbits
    dev = tgt_codes.device
    if idx is None:
        idx = torch.empty(n_tgt, dtype=torch.int32, device=dev)
    if dist is None:
        dist = torch.empty(n_tgt, dtype=torch.int32, device=dev)
    if workspace is None:
        workspace = torch.empty(max(256, semshare_match_tc_workspace_size(n_tgt, n_ref, nbits)), dtype=torch.uint8,
                                device=dev)
    args = (_ptr(tgt_codes), n_tgt, _ptr(ref_codes), n_ref, nbits, _ptr(idx), _ptr(dist), _ptr(workspace),
            workspace.numel() * workspace.element_size(), _ptr(err_flag))
    call = Prepared(load().semshare_match_tc, args, "semshare_match_tc", (tgt_codes, ref_codes, workspace, err_flag),
                    (idx, dist))
    return call if prepare else call(stream)


_match_signs_ws = {}
# Targets up to which semshare_match_tc_signs is one launch (include/semshare.h); above it a small
# split launch follows the search.
MATCH_SIGNS_FUSED_MAX_TARGETS = 16384


def semshare_match_tc_signs_workspace_size(n_tgt: int) -> int:
    return int(load().semshare_match_tc_signs_workspace_size(int(n_tgt)))


def match_signs_workspace(n_tgt: int, device=None) -> torch.Tensor:
    """A 0xFF-filled semshare_match_tc_signs workspace large enough for n_tgt targets, kept per
    device and grown on demand.  Every call leaves it 0xFF-filled, so calls issued one after
    another (on one stream) can share it; concurrent calls need their own."""
    dev = torch.device(device or "cuda")
    if dev.index is None:
        dev = torch.device("cuda", torch.cuda.current_device())
    need = max(512, semshare_match_tc_signs_workspace_size(n_tgt))
    ws = _match_signs_ws.get(dev)
    if ws is None or ws.numel() < need:
        ws = torch.full((need,), 0xFF, dtype=torch.uint8, device=dev)
        _match_signs_ws[dev] = ws
    return ws


def semshare_match_tc_signs(tgt_signs: torch.Tensor, ref_signs: torch.Tensor, nbits: int,
                            idx: torch.Tensor | None = None, dist: torch.Tensor | None = None,
                            workspace: torch.Tensor | None = None, err_flag: torch.Tensor | None = None,
                            stream=None, *, prepare: bool = False):
    """semshare_match_tc on the sign rows of semshare_hash_signs (uint8 [n][pitch], rows may be a
    slice of one hash call's output), in one launch.  workspace: 0xFF-filled (default: the
    per-device one of match_signs_workspace()).  Returns (idx, dist)."""
    _need_cuda(tgt_signs, "tgt_signs")
    _need_cuda(ref_signs, "ref_signs")
    pitch = semshare_signs_pitch(nbits)
    for name, t in (("tgt_signs", tgt_signs), ("ref_signs", ref_signs)):
        if t.dtype != torch.uint8 or t.dim() != 2 or t.shape[1] != pitch or not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous uint8 [n][{pitch}]")
    n_tgt, n_ref = tgt_signs.shape[0], ref_signs.shape[0]
    dev = tgt_signs.device
    if idx is None:
        idx = torch.empty(n_tgt, dtype=torch.int32, device=dev)
    if dist is None:
        dist = torch.empty(n_tgt, dtype=torch.int32, device=dev)
    if workspace is None:
        workspace = match_signs_workspace(n_tgt, dev)
    args = (_ptr(tgt_signs), n_tgt, _ptr(ref_signs), n_ref, int(nbits), _ptr(idx), _ptr(dist), _ptr(workspace),
            workspace.numel() * workspace.element_size(), _ptr(err_flag))
    call = Prepared(load().semshare_match_tc_signs, args, "semshare_match_tc_signs",
                    (tgt_signs, ref_signs, workspace, err_flag), (idx, dist))
    return call if prepare else call(stream)


RETRIEVE_MAX_CANDIDATES = 256
SIMILARITY_MAX_DIST = 30.0   # App. A.3: max(dist) of the normalised LSH distance
SIMILARITY_THRESHOLD = 0.8   # Sec. 4.4: reuse applies above this similarity


def semshare_retrieve_workspace_size(n_tgt: int, n_pool: int, n_cand: int, nbits: int) -> int:
    return int(load().semshare_retrieve_workspace_size(int(n_tgt), int(n_pool), int(n_cand), int(nbits)))


class Retrieval(NamedTuple):
    """Outputs of semshare_retrieve, all device tensors."""
    mean_dist: torch.Tensor   # float64 [n_cand]: LSH_dist of every candidate
    similarity: torch.Tensor  # float64 [n_cand]
    best: torch.Tensor        # int32 [1]: candidate of greatest similarity
    applies: torch.Tensor     # int32 [1]: 1 if similarity[best] > threshold
    idx: torch.Tensor | None  # int32 [n_tgt]: nearest global pool row within the best candidate
    dist: torch.Tensor | None


def semshare_retrieve(tgt_codes: torch.Tensor, pool_codes: torch.Tensor, cand_offsets,
                      max_dist: float = SIMILARITY_MAX_DIST, threshold: float = SIMILARITY_THRESHOLD,
                      want_match: bool = True, workspace: torch.Tensor | None = None,
                      err_flag: torch.Tensor | None = None, nbits: int | None = None, stream=None,
                      out: Retrieval | None = None) -> Retrieval:
    """Reference retrieval by LSH-distance similarity (Sec. 3.2, App. A.3, Sec. 4.4).

    pool_codes holds the candidates' codes back to back; cand_offsets (host sequence of
    n_cand + 1 ints) delimits them.  With want_match, idx/dist are the nearest rows of the
    best candidate for every target row.  `out` (a Retrieval of preallocated device tensors,
    idx/dist None to skip the match) is filled instead of allocating."""
    _need_cuda(tgt_codes, "tgt_codes")
    _need_cuda(pool_codes, "pool_codes")
    if not tgt_codes.is_contiguous() or not pool_codes.is_contiguous():
        raise ValueError("codes must be contiguous")
    n_tgt, w = tgt_codes.shape
    if pool_codes.shape[1] != w:
        raise ValueError("code widths differ")
    offs = (ctypes.c_int64 * len(cand_offsets))(*[int(o) for o in cand_offsets])
    n_cand = len(cand_offsets) - 1
    nbits = 32 * w if nbits is None else nbits
    dev = tgt_codes.device
    if out is not None:
        mean, sim, best, applies, idx, dist = out
        for t, n in ((mean, n_cand), (sim, n_cand), (best, 1), (applies, 1), (idx, n_tgt), (dist, n_tgt)):
            if t is not None and (t.device != dev or not t.is_contiguous() or t.numel() < n):
                raise ValueError("preallocated retrieval output of the wrong size or device")
    else:
        mean = torch.empty(max(n_cand, 1), dtype=torch.float64, device=dev)
        sim = torch.empty(max(n_cand, 1), dtype=torch.float64, device=dev)
        choice = torch.empty(2, dtype=torch.int32, device=dev)
        best, applies = choice[:1], choice[1:]
        idx = dist = None
        if want_match:
            idx = torch.empty(n_tgt, dtype=torch.int32, device=dev)
            dist = torch.empty(n_tgt, dtype=torch.int32, device=dev)
    if workspace is None:
        need = semshare_retrieve_workspace_size(n_tgt, int(pool_codes.shape[0]), n_cand, nbits)
        workspace = torch.empty(max(256, need), dtype=torch.uint8, device=dev)
    st = load().semshare_retrieve(_ptr(tgt_codes), n_tgt, _ptr(pool_codes), offs, n_cand, nbits, float(max_dist),
                                  float(threshold), _ptr(mean), _ptr(sim), _ptr(best), _ptr(applies),
                                  _ptr(idx), _ptr(dist), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                  _ptr(err_flag), _stream(stream))
    _check(st, "semshare_retrieve")
    if out is not None:
        return out
    return Retrieval(mean[:n_cand], sim[:n_cand], best, applies, idx, dist)


def semshare_match_tc_selected_workspace_size(n_tgt: int, cand_offsets, nbits: int) -> int:
    offs = (ctypes.c_int64 * len(cand_offsets))(*[int(o) for o in cand_offsets])
    return int(load().semshare_match_tc_selected_workspace_size(int(n_tgt), offs, len(cand_offsets) - 1, int(nbits)))


def semshare_match_tc_selected(tgt_codes: torch.Tensor, pool_codes: torch.Tensor, cand_offsets, best: torch.Tensor,
                               idx: torch.Tensor | None = None, dist: torch.Tensor | None = None,
                               workspace: torch.Tensor | None = None, err_flag: torch.Tensor | None = None,
                               nbits: int | None = None, stream=None):
    """Token matching (Sec. 3.3) against candidate `best` (a device int32, e.g. the retrieval's
    choice) of the pool delimited by cand_offsets, read on the device: no host round trip.
    Returns (idx, dist) int32 [n_tgt] with idx in pool rows."""
    for t, n in ((tgt_codes, "tgt_codes"), (pool_codes, "pool_codes"), (best, "best")):
        _need_cuda(t, n)
    if not tgt_codes.is_contiguous() or not pool_codes.is_contiguous():
        raise ValueError("codes must be contiguous")
    if best.dtype != torch.int32:
        raise ValueError("best must be int32")
    n_tgt, w = tgt_codes.shape
    if pool_codes.shape[1] != w:
        raise ValueError("code widths differ")
    nbits = 32 * w if nbits is None else nbits
    offs = (ctypes.c_int64 * len(cand_offsets))(*[int(o) for o in cand_offsets])
    n_cand = len(cand_offsets) - 1
    dev = tgt_codes.device
    if idx is None:
        idx = torch.empty(n_tgt, dtype=torch.int32, device=dev)
    if dist is None:
        dist = torch.empty(n_tgt, dtype=torch.int32, device=dev)
    _need_cuda(idx, "idx")
    _need_cuda(dist, "dist")
    if workspace is None:
        need = semshare_match_tc_selected_workspace_size(n_tgt, cand_offsets, nbits)
        workspace = torch.empty(max(256, need), dtype=torch.uint8, device=dev)
    st = load().semshare_match_tc_selected(_ptr(tgt_codes), n_tgt, _ptr(pool_codes), offs, n_cand, _ptr(best), nbits,
                                           _ptr(idx), _ptr(dist), _ptr(workspace),
                                           workspace.numel() * workspace.element_size(), _ptr(err_flag),
                                           _stream(stream))
    _check(st, "semshare_match_tc_selected")
    return idx, dist


def semshare_match_static(tgt_codes: torch.Tensor, ref_codes: torch.Tensor, idx: torch.Tensor | None = None,
                          dist: torch.Tensor | None = None, nbits: int | None = None, stream=None):
    """semshare_match for callers that cannot allocate device memory: no workspace argument,
    the library's own fixed scratch (at most MATCH_STATIC_MAX_TARGETS targets) is used.
    Pass preallocated idx/dist to keep the call itself free of allocations.
    Returns (idx int32 [n_tgt], dist int32 [n_tgt])."""
    _need_cuda(tgt_codes, "tgt_codes")
    _need_cuda(ref_codes, "ref_codes")
    if not tgt_codes.is_contiguous() or not ref_codes.is_contiguous():
        raise ValueError("codes must be contiguous")
    n_tgt, w = tgt_codes.shape
    if ref_codes.shape[1] != w:
        raise ValueError("code widths differ")
    nbits = 32 * w if nbits is None else nbits
    if idx is None:
        idx = torch.empty(n_tgt, dtype=torch.int32, device=tgt_codes.device)
    if dist is None:
        dist = torch.empty(n_tgt, dtype=torch.int32, device=tgt_codes.device)
    st = load().semshare_match_static(_ptr(tgt_codes), n_tgt, _ptr(ref_codes), ref_codes.shape[0], nbits, _ptr(idx),
                                      _ptr(dist), _stream(stream))
    _check(st, "semshare_match_static")
    return idx, dist


def kv_layout(t: torch.Tensor, batched: bool) -> KVLayout:
    """Layout of a [B][L][H][T][hd] (batched) or [L][H][T][hd] cache tensor."""
    if t.stride(-1) != 1:
        raise ValueError("head_dim must be contiguous")
    if batched:
        if t.dim() != 5:
            raise ValueError("expected [n_batch][L][H][T][head_dim]")
        sb, sl, sh, st = t.stride(0), t.stride(1), t.stride(2), t.stride(3)
        L, H, hd = t.shape[1], t.shape[2], t.shape[4]
    else:
        if t.dim() != 4:
            raise ValueError("expected [L][H][T][head_dim]")
        sb, (sl, sh, st) = 0, t.stride()[:3]
        L, H, hd = t.shape[0], t.shape[1], t.shape[3]
    return KVLayout(L, H, hd, t.element_size(), sb, sl, sh, st)


def _segments(ref_k, ref_v):
    """The K and V segments of a reference cache (a tensor or a list of tensors sharing one layout),
    checked: CUDA or pinned host, [L][H][N][hd] with head_dim contiguous, one layout throughout.
    Returns (seg_k, seg_v, layout of the first segment)."""
    seg_k = ref_k if isinstance(ref_k, (list, tuple)) else (ref_k,)
    seg_v = ref_v if isinstance(ref_v, (list, tuple)) else (ref_v,)
    if len(seg_k) != len(seg_v) or not seg_k:
        raise ValueError("ref_k and ref_v must have the same number of segments")
    k0 = seg_k[0]
    src = kv_layout(k0, batched=False)
    key = (k0.stride()[:3], k0.shape[0], k0.shape[1], k0.shape[3], k0.element_size())
    for t in (*seg_k, *seg_v):
        _need_device_accessible(t, "ref")
        if t.dim() != 4 or t.stride(3) != 1 or (t.stride()[:3], t.shape[0], t.shape[1], t.shape[3],
                                                  t.element_size()) != key:
            raise ValueError("all segments must share one layout")
    return seg_k, seg_v, src


def semshare_gather_kv(ref_k, ref_v, idx: torch.Tensor, out_k: torch.Tensor | None = None,
                       out_v: torch.Tensor | None = None, err_flag: torch.Tensor | None = None, stream=None, *,
                       prepare: bool = False):
    """Reordered K/V cache: out[b][l][h][t] = ref[l][h][idx[b][t]].

    ref_k/ref_v: a [L][H][N][hd] CUDA or pinned host tensor, or a list of them (a pool of reference prompts
    with identical strides; global row r = running offset of its segment + local row).
    idx: [n_batch][n_tgt] or [n_tgt] int32.  Returns (out_k, out_v), [n_batch][L][H][n_tgt][hd]."""
    seg_k, seg_v, src = _segments(ref_k, ref_v)
    _need_cuda(idx, "idx")
    idx2 = idx if idx.dim() == 2 else idx.view(1, -1)
    if idx2.dtype != torch.int32 or not idx2.is_contiguous():
        raise ValueError("idx must be contiguous int32")
    n_batch, n_tgt = idx2.shape
    L, H, hd = src.n_layers, src.n_heads, src.head_dim
    if out_k is None:
        out_k = torch.empty((n_batch, L, H, n_tgt, hd), dtype=seg_k[0].dtype, device=idx.device)
    if out_v is None:
        out_v = torch.empty((n_batch, L, H, n_tgt, hd), dtype=seg_v[0].dtype, device=idx.device)
    _need_cuda(out_k, "out_k")
    _need_cuda(out_v, "out_v")
    dst = kv_layout(out_k, batched=True)
    if out_v.dim() != 5 or out_v.stride() != out_k.stride():
        raise ValueError("out_k and out_v must share one layout")
    n_seg = len(seg_k)
    if n_seg == 1:
        pk = (ctypes.c_void_p * 1)(seg_k[0].data_ptr())
        pv = (ctypes.c_void_p * 1)(seg_v[0].data_ptr())
        po = (ctypes.c_int64 * 2)(0, seg_k[0].shape[2])
    else:
        offs = [0]
        for t in seg_k:
            offs.append(offs[-1] + t.shape[2])
        pk = (ctypes.c_void_p * n_seg)(*[t.data_ptr() for t in seg_k])
        pv = (ctypes.c_void_p * n_seg)(*[t.data_ptr() for t in seg_v])
        po = (ctypes.c_int64 * (n_seg + 1))(*offs)
    args = (pk, pv, po, n_seg, src, _ptr(idx2), n_tgt, n_batch, _ptr(out_k), _ptr(out_v), dst, _ptr(err_flag))
    call = Prepared(load().semshare_gather_kv, args, "semshare_gather_kv", (seg_k, seg_v, idx2, err_flag),
                    (out_k, out_v))
    return call if prepare else call(stream)


def semshare_fetch_workspace_size(n_rows: int) -> int:
    return int(load().semshare_fetch_workspace_size(int(n_rows)))


def semshare_fetch_rows(ref_k, ref_v, idx: torch.Tensor, dev_k=None, dev_v=None, workspace: torch.Tensor | None = None,
                        err_flag: torch.Tensor | None = None, stream=None):
    """Copies the reference rows idx selects -- each once, whatever its count in idx -- from
    ref_k/ref_v (CUDA or pinned host tensors [L][H][N][hd], or lists of them sharing one layout)
    into device caches dev_k/dev_v of the same shapes and strides (allocated on idx.device when
    None).  Rows no idx names are left as they were.  Returns (dev_k, dev_v), lists when the
    sources are lists; semshare_gather_kv on them with the same idx gives the gather of the
    sources."""
    as_list = isinstance(ref_k, (list, tuple))
    seg_k, seg_v, lay = _segments(ref_k, ref_v)
    seg_k, seg_v = list(seg_k), list(seg_v)
    _need_cuda(idx, "idx")
    if idx.dtype != torch.int32 or not idx.is_contiguous():
        raise ValueError("idx must be contiguous int32")

    def like(ts):
        return [torch.empty_strided(t.shape, t.stride(), dtype=t.dtype, device=idx.device) for t in ts]

    dk = like(seg_k) if dev_k is None else (list(dev_k) if isinstance(dev_k, (list, tuple)) else [dev_k])
    dv = like(seg_v) if dev_v is None else (list(dev_v) if isinstance(dev_v, (list, tuple)) else [dev_v])
    if len(dk) != len(seg_k) or len(dv) != len(seg_v):
        raise ValueError("dev_k/dev_v need one tensor per segment")
    for d, t in zip(dk + dv, seg_k + seg_v):
        _need_cuda(d, "dev")
        if d.shape != t.shape or d.stride() != t.stride() or d.dtype != t.dtype:
            raise ValueError("dev_k/dev_v must have the shapes, strides and dtype of ref_k/ref_v")
    n_seg = len(seg_k)
    offs = [0]
    for t in seg_k:
        offs.append(offs[-1] + t.shape[2])
    if workspace is None:
        workspace = torch.empty(max(semshare_fetch_workspace_size(offs[-1]), 16), dtype=torch.uint8,
                                device=idx.device)
    _need_cuda(workspace, "workspace")
    arr = lambda ts: (ctypes.c_void_p * n_seg)(*[t.data_ptr() for t in ts])  # noqa: E731
    po = (ctypes.c_int64 * (n_seg + 1))(*offs)
    st = load().semshare_fetch_rows(arr(seg_k), arr(seg_v), arr(dk), arr(dv), po, n_seg, lay, _ptr(idx), idx.numel(),
                                    _ptr(workspace), workspace.numel() * workspace.element_size(), _ptr(err_flag),
                                    _stream(stream))
    _check(st, "semshare_fetch_rows")
    return (dk, dv) if as_list else (dk[0], dv[0])


HD_PERCENT = 40  # Insight 1: the 40% of tokens with the highest deviation are HD tokens


def hd_count(n_tok: int, percent: int = HD_PERCENT) -> int:
    """Number of HD tokens, ceil(percent% of n_tok) (semshare_hd_count)."""
    k = int(load().semshare_hd_count(int(n_tok), int(percent)))
    if k < 0:
        raise SemshareError(EINVAL, "semshare_hd_count")
    return k


def semshare_kv_deviation(k_reused: torch.Tensor, v_reused: torch.Tensor, k_recomp: torch.Tensor,
                          v_recomp: torch.Tensor, sigma_kv: torch.Tensor | None = None,
                          sigma_k: torch.Tensor | None = None, sigma_v: torch.Tensor | None = None,
                          want_parts: bool = False, stream=None):
    """Key-Value deviation (App. A.4) per layer and token of [L][H][T][hd] caches (bf16 or fp32;
    strided views allowed, head_dim contiguous).  Returns sigma_kv, or (sigma_k, sigma_v,
    sigma_kv) with want_parts; each float32 [L][T]."""
    ts = (k_reused, v_reused, k_recomp, v_recomp)
    for t, n in zip(ts, ("k_reused", "v_reused", "k_recomp", "v_recomp")):
        _need_cuda(t, n)
    if k_reused.dtype == torch.bfloat16:
        dt = BF16
    elif k_reused.dtype == torch.float32:
        dt = F32
    else:
        raise TypeError("caches must be bfloat16 or float32")
    if any(t.dtype != k_reused.dtype or t.shape != k_reused.shape for t in ts) or k_reused.dim() != 4:
        raise ValueError("four [L][H][T][hd] caches of one shape and dtype")
    if v_reused.stride() != k_reused.stride() or v_recomp.stride() != k_recomp.stride():
        raise ValueError("K and V of a cache must share strides")
    L, _, T, _ = k_reused.shape
    dev = k_reused.device
    if sigma_kv is None:
        sigma_kv = torch.empty((L, T), dtype=torch.float32, device=dev)
    if want_parts:
        sigma_k = torch.empty((L, T), dtype=torch.float32, device=dev) if sigma_k is None else sigma_k
        sigma_v = torch.empty((L, T), dtype=torch.float32, device=dev) if sigma_v is None else sigma_v
    st = load().semshare_kv_deviation(_ptr(k_reused), _ptr(v_reused), kv_layout(k_reused, False), _ptr(k_recomp),
                                      _ptr(v_recomp), kv_layout(k_recomp, False), dt, T, _ptr(sigma_k),
                                      _ptr(sigma_v), _ptr(sigma_kv), _stream(stream))
    _check(st, "semshare_kv_deviation")
    return (sigma_k, sigma_v, sigma_kv) if want_parts else sigma_kv


def semshare_select_hd(sigma: torch.Tensor, k: int | None = None, hd_idx: torch.Tensor | None = None,
                       want_mask: bool = False, hd_mask: torch.Tensor | None = None, stream=None):
    """The k highest-deviation tokens of every layer (default k = hd_count(T)), ascending, ties
    to the lower index.  sigma: float32 [L][T] (or [T]).  Returns hd_idx int32 [L][k] (and the
    uint8 [L][T] mask with want_mask)."""
    _need_cuda(sigma, "sigma")
    if sigma.dtype != torch.float32 or not sigma.is_contiguous():
        raise ValueError("sigma must be a contiguous float32 tensor")
    s2 = sigma.view(1, -1) if sigma.dim() == 1 else sigma
    L, T = s2.shape
    k = hd_count(T) if k is None else int(k)
    if hd_idx is None:
        hd_idx = torch.empty((L, k), dtype=torch.int32, device=sigma.device)
    if want_mask and hd_mask is None:
        hd_mask = torch.empty((L, T), dtype=torch.uint8, device=sigma.device)
    st = load().semshare_select_hd(_ptr(s2), L, T, k, _ptr(hd_idx), _ptr(hd_mask), _stream(stream))
    _check(st, "semshare_select_hd")
    return (hd_idx, hd_mask) if want_mask else hd_idx


RETAIN_MAX_LAYERS = 128


def retain_counts(n_tok: int, alpha_num, alpha_den: int) -> list:
    """Retained tokens per layer, Retain[i] = floor(T * prod_{j<=i} alpha_num[j] / alpha_den)
    (App. A), computed exactly by semshare_retain_counts."""
    num = [int(a) for a in alpha_num]
    n = len(num)
    arr = (ctypes.c_int32 * max(n, 1))(*num)
    out = (ctypes.c_int64 * max(n, 1))()
    _check(load().semshare_retain_counts(int(n_tok), arr, int(alpha_den), n, out), "semshare_retain_counts")
    return [int(out[i]) for i in range(n)]


def semshare_gather_kv_retained(ref_k, ref_v, idx: torch.Tensor, retained, ret_offsets,
                                out_k: torch.Tensor | None = None, out_v: torch.Tensor | None = None,
                                err_flag: torch.Tensor | None = None, stream=None):
    """Retention-aware rearrangement (Sec. 3.3.4): out[l][h][r] = ref[l][h][idx[retained_l[r]]].

    ref_k/ref_v: a [L][H][N][hd] CUDA or pinned host tensor, or a list of them (as semshare_gather_kv).
    idx: int32 [n_tgt].  retained: int32 CUDA tensor, the layers' lists back to back;
    ret_offsets: host sequence of L + 1 ints.  Returns (out_k, out_v), [L][H][longest][hd]."""
    seg_k, seg_v, src = _segments(ref_k, ref_v)
    _need_cuda(idx, "idx")
    _need_cuda(retained, "retained")
    if idx.dtype != torch.int32 or not idx.is_contiguous() or retained.dtype != torch.int32 or \
            not retained.is_contiguous():
        raise ValueError("idx and retained must be contiguous int32")
    L, H, hd = src.n_layers, src.n_heads, src.head_dim
    if len(ret_offsets) != L + 1:
        raise ValueError("ret_offsets needs n_layers + 1 entries")
    longest = max(int(ret_offsets[l + 1]) - int(ret_offsets[l]) for l in range(L))
    if out_k is None:
        out_k = torch.empty((L, H, max(longest, 0), hd), dtype=seg_k[0].dtype, device=idx.device)
    if out_v is None:
        out_v = torch.empty((L, H, max(longest, 0), hd), dtype=seg_v[0].dtype, device=idx.device)
    _need_cuda(out_k, "out_k")
    _need_cuda(out_v, "out_v")
    dst = kv_layout(out_k, batched=False)
    if kv_layout(out_v, batched=False).stride_token != dst.stride_token or out_v.stride() != out_k.stride():
        raise ValueError("out_k and out_v must share one layout")
    offs = [0]
    for t in seg_k:
        offs.append(offs[-1] + t.shape[2])
    n_seg = len(seg_k)
    pk = (ctypes.c_void_p * n_seg)(*[t.data_ptr() for t in seg_k])
    pv = (ctypes.c_void_p * n_seg)(*[t.data_ptr() for t in seg_v])
    po = (ctypes.c_int64 * (n_seg + 1))(*offs)
    ro = (ctypes.c_int64 * (L + 1))(*[int(o) for o in ret_offsets])
    st = load().semshare_gather_kv_retained(pk, pv, po, n_seg, src, _ptr(idx), idx.numel(), _ptr(retained), ro,
                                            _ptr(out_k), _ptr(out_v), dst, _ptr(err_flag), _stream(stream))
    _check(st, "semshare_gather_kv_retained")
    return out_k, out_v

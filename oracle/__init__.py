"""CPU oracle for the fuzzy token-matching path -- TEST INFRASTRUCTURE ONLY.

Only `tests/`, `__graft_entry__.smoke()` and the CPU-baseline leg of `bench.py` may import
this package.  It wraps `semshare_oracle.c` (plain C, fp64, OpenMP over rows) with numpy
in/out arrays.  It shares no code with the CUDA library and never imports it.

What each function computes, and the passage of the paper (SemShareKV, arXiv 2509.24832)
it follows, is stated in `semshare_oracle.c`:
  rope    Eq. 1 (App. A.1) with angle m*theta_k; Sec. 3.3.1
  hash    random-hyperplane sign codes of the rotated rows; Sec. 3.3, App. A.2
  match   Hamming 1-nearest reference token, ties to the lowest index; Sec. 3.3
  gather  reordered K/V rows, bitwise copies; Sec. 3.3, Sec. 3.3.2
  retrieve  LSH-distance similarity of whole prompts and the best candidate; Sec. 3.2,
          App. A.3, Sec. 4.4
  kv_deviation  sigma_K + sigma_V per layer and token; App. A.4
  select_hd     the k highest-deviation tokens per layer; Insight 1, Sec. 3.2
  gather_kv_retained  the rearranged rows of each layer's retained tokens only; Sec. 3.3.4, App. A
  fetch_rows    the reference rows the match selects, loaded once each; Sec. 3.2, Sec. 3.3

Parity pins: every function here is pinned by `tests/test_oracle_*.py` against closed forms,
invariants, hand-derived golden cases and brute force (none is "parity unpinned").
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "semshare_oracle.c")
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIBDIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

_CFLAGS = ["-O2", "-fopenmp", "-ffp-contract=off", "-fno-fast-math", "-shared", "-fPIC", "-std=c11"]


def build(force: bool = False) -> str:
    """Compile the oracle with gcc into oracle/_lib/liboracle.so (no-op when up to date)."""
    os.makedirs(_LIBDIR, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.run(["gcc", *_CFLAGS, _SRC, "-o", tmp, "-lm"], check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        lib.oracle_num_threads.restype = ctypes.c_int
        lib.oracle_set_threads.argtypes = [ctypes.c_int]
        lib.oracle_set_threads.restype = ctypes.c_int
        lib.oracle_bf16_value.argtypes = [ctypes.c_uint16]
        lib.oracle_bf16_value.restype = f64
        lib.oracle_bf16_round.argtypes = [f64]
        lib.oracle_bf16_round.restype = ctypes.c_uint16
        lib.oracle_theta.argtypes = [i32, i32, f64]
        lib.oracle_theta.restype = f64
        lib.oracle_rope.argtypes = [P, i64, i32, P, f64, P]
        lib.oracle_rope_layout.argtypes = [P, i64, i32, P, f64, P, i32]
        lib.oracle_hash.argtypes = [P, i32, i64, i32, i64, P, f64, P, i32, P, P, i32]
        lib.oracle_hash_layout.argtypes = [P, i32, i64, i32, i64, P, f64, P, i32, P, P, i32, i32]
        lib.oracle_hamming.argtypes = [P, P, i32]
        lib.oracle_hamming.restype = i32
        lib.oracle_match.argtypes = [P, i64, P, i64, i32, P, P]
        lib.oracle_gather_kv.argtypes = [P, P, P, i32, i32, i32, i64, P, i64, i32, P, P]
        lib.oracle_gather_kv.restype = i64
        lib.oracle_retrieve.argtypes = [P, i64, P, P, i32, i32, f64, f64, P, P, P, P]
        lib.oracle_kv_deviation.argtypes = [P, P, P, P, i32, i32, i32, i64, i32, P, P, P]
        lib.oracle_select_hd.argtypes = [P, i32, i64, i64, P]
        lib.oracle_gather_kv_retained.argtypes = [P, P, i32, i32, i64, i64, P, i64, P, P, i64, P, P]
        lib.oracle_gather_kv_retained.restype = i64
        lib.oracle_fetch_rows.argtypes = [P, P, P, P, P, i32, i32, i32, i64, P, i64]
        lib.oracle_fetch_rows.restype = i64
        _lib = lib
        return lib


def _ptr(a: np.ndarray | None):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def num_threads() -> int:
    """OpenMP threads the oracle uses (OMP_NUM_THREADS, else all cores)."""
    return int(_load().oracle_num_threads())


def set_threads(n: int) -> int:
    """Sets the OpenMP threads of the oracle's later calls; returns the previous count (timing only:
    the results do not depend on it)."""
    return int(_load().oracle_set_threads(int(n)))


def bf16_round(v: float) -> int:
    """Nearest bf16 bit pattern to the fp64 value v (ties to even)."""
    return int(_load().oracle_bf16_round(float(v)))


def bf16_value(h: int) -> float:
    return float(_load().oracle_bf16_value(int(h)))


def theta(k: int, d: int, base: float = 10000.0) -> float:
    """Rotation frequency theta_k = base^(-2k/d) of pair k (Eq. 1)."""
    return float(_load().oracle_theta(k, d, base))


LAYOUTS = {"interleaved": 0, "half": 1}


def rope(x: np.ndarray, positions, base: float = 10000.0, layout: str = "interleaved") -> np.ndarray:
    """fp64 rotary encoding of rows x[n][d] at the given positions (Eq. 1, Sec. 3.3.1); pairs
    (2k, 2k+1) as Eq. 1 prints them, or (k, k + d/2) with layout="half"."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    n, d = x.shape
    pos = np.ascontiguousarray(np.broadcast_to(np.asarray(positions, dtype=np.int32), (n,)))
    y = np.empty_like(x)
    _load().oracle_rope_layout(_ptr(x), n, d, _ptr(pos), base, _ptr(y), LAYOUTS[layout])
    return y


def hash_codes(emb: np.ndarray, positions, hyperplanes: np.ndarray, base: float = 10000.0,
               round_operand: bool = True, layout: str = "interleaved"):
    """LSH codes of embedding rows (Sec. 3.3, App. A.2).

    emb: [n][d] float32 rows, or uint16 bf16 bit patterns.  hyperplanes: [nbits][d] uint16 bf16.
    Returns (codes [n][nbits/32] uint32, proj [n][nbits] float32)."""
    emb = np.ascontiguousarray(emb)
    if emb.dtype == np.float32:
        f32 = 1
    elif emb.dtype == np.uint16:
        f32 = 0
    else:
        raise TypeError("emb must be float32 or bf16 bit patterns (uint16)")
    n, d = emb.shape
    R = np.ascontiguousarray(hyperplanes, dtype=np.uint16)
    nbits = R.shape[0]
    if R.shape[1] != d or nbits % 32 or d % 2:
        raise ValueError("shape mismatch")
    pos = None if positions is None else np.ascontiguousarray(np.asarray(positions, dtype=np.int32).reshape(n))
    codes = np.zeros((n, nbits // 32), dtype=np.uint32)
    proj = np.zeros((n, nbits), dtype=np.float32)
    _load().oracle_hash_layout(_ptr(emb), f32, n, d, d, _ptr(pos), base, _ptr(R), nbits, _ptr(codes), _ptr(proj),
                               1 if round_operand else 0, LAYOUTS[layout])
    return codes, proj


def hamming(a: np.ndarray, b: np.ndarray) -> int:
    a = np.ascontiguousarray(a, dtype=np.uint32)
    b = np.ascontiguousarray(b, dtype=np.uint32)
    return int(_load().oracle_hamming(_ptr(a), _ptr(b), a.shape[-1]))


def match(tgt_codes: np.ndarray, ref_codes: np.ndarray, nbits: int | None = None):
    """Hamming 1-nearest reference row of every target row, ties to the lowest index (Sec. 3.3).

    Returns (idx int32 [n_tgt], dist int32 [n_tgt])."""
    t = np.ascontiguousarray(tgt_codes, dtype=np.uint32)
    r = np.ascontiguousarray(ref_codes, dtype=np.uint32)
    w = t.shape[1]
    nbits = 32 * w if nbits is None else nbits
    idx = np.empty(t.shape[0], dtype=np.int32)
    dist = np.empty(t.shape[0], dtype=np.int32)
    _load().oracle_match(_ptr(t), t.shape[0], _ptr(r), r.shape[0], nbits, _ptr(idx), _ptr(dist))
    return idx, dist


def gather_kv(seg_k, seg_v, idx: np.ndarray, out_k: np.ndarray | None = None, out_v: np.ndarray | None = None):
    """Reordered KV cache (Sec. 3.3): out[b][l][h][t] = ref[l][h][idx[b][t]].

    seg_k/seg_v: one array [L][H][n_s][hd] per reference segment (a list, or a single array for
    one reference).  Global reference row r of segment s is local row r - offset[s], offsets
    being the running sum of the n_s.  idx: [n_batch][n_tgt] (or [n_tgt]).
    Returns (out_k, out_v, n_bad) with out [n_batch][L][H][n_tgt][hd]; rows with an out-of-range
    idx are left as they were in out_k/out_v (zeros when allocated here) and counted in n_bad."""
    if isinstance(seg_k, np.ndarray):
        seg_k, seg_v = [seg_k], [seg_v]
    seg_k = [np.ascontiguousarray(a) for a in seg_k]
    seg_v = [np.ascontiguousarray(a) for a in seg_v]
    L, H, _, hd = seg_k[0].shape
    dt = seg_k[0].dtype
    idx2 = np.ascontiguousarray(np.atleast_2d(np.asarray(idx, dtype=np.int32)))
    B, n_tgt = idx2.shape
    offs = np.zeros(len(seg_k) + 1, dtype=np.int64)
    for s, a in enumerate(seg_k):
        if a.shape[:2] != (L, H) or a.shape[3] != hd or seg_v[s].shape != a.shape:
            raise ValueError("segment shapes differ")
        offs[s + 1] = offs[s] + a.shape[2]
    if out_k is None:
        out_k = np.zeros((B, L, H, n_tgt, hd), dtype=dt)
    if out_v is None:
        out_v = np.zeros((B, L, H, n_tgt, hd), dtype=dt)
    pk = (ctypes.c_void_p * len(seg_k))(*[a.ctypes.data for a in seg_k])
    pv = (ctypes.c_void_p * len(seg_v))(*[a.ctypes.data for a in seg_v])
    bad = _load().oracle_gather_kv(pk, pv, _ptr(offs), len(seg_k), L, H, hd * dt.itemsize, _ptr(idx2), n_tgt, B,
                                   _ptr(out_k), _ptr(out_v))
    return out_k, out_v, int(bad)


def retrieve(tgt_codes: np.ndarray, pool_codes: np.ndarray, seg_offsets, nbits: int | None = None,
             max_dist: float = 30.0, threshold: float = 0.8):
    """Reference retrieval by LSH-distance similarity (Sec. 3.2, App. A.3, Sec. 4.4).

    pool_codes: the candidate prompts' codes concatenated; candidate s is rows
    seg_offsets[s]..seg_offsets[s+1].  Returns (mean_dist [n_seg] float64, similarity [n_seg]
    float64, best, applies)."""
    t = np.ascontiguousarray(tgt_codes, dtype=np.uint32)
    p = np.ascontiguousarray(pool_codes, dtype=np.uint32)
    offs = np.ascontiguousarray(np.asarray(seg_offsets, dtype=np.int64))
    n_seg = len(offs) - 1
    nbits = 32 * t.shape[1] if nbits is None else nbits
    mean = np.zeros(n_seg)
    sim = np.zeros(n_seg)
    best = np.zeros(1, dtype=np.int32)
    applies = np.zeros(1, dtype=np.int32)
    _load().oracle_retrieve(_ptr(t), t.shape[0], _ptr(p), _ptr(offs), n_seg, nbits, float(max_dist), float(threshold),
                            _ptr(mean), _ptr(sim), _ptr(best), _ptr(applies))
    return mean, sim, int(best[0]), bool(applies[0])


def kv_deviation(k_re, v_re, k_rc, v_rc):
    """Key-Value deviation (App. A.4) of [L][H][T][hd] arrays (bf16 bit patterns as uint16, or
    float32): returns (sigma_k, sigma_v, sigma_kv), each [L][T] float64."""
    arrs = [np.ascontiguousarray(a) for a in (k_re, v_re, k_rc, v_rc)]
    dt = arrs[0].dtype
    if dt not in (np.uint16, np.float32) or any(a.dtype != dt or a.shape != arrs[0].shape for a in arrs):
        raise ValueError("four [L][H][T][hd] arrays of one dtype (uint16 bf16 bits or float32)")
    L, H, T, hd = arrs[0].shape
    sk = np.zeros((L, T))
    sv = np.zeros((L, T))
    skv = np.zeros((L, T))
    _load().oracle_kv_deviation(*[_ptr(a) for a in arrs], 1 if dt == np.float32 else 0, L, H, T, hd, _ptr(sk),
                                _ptr(sv), _ptr(skv))
    return sk, sv, skv


def select_hd(sigma, k: int):
    """The k highest-deviation tokens of every layer (ties to the lower index), ascending:
    sigma [L][T] (any float type; taken as float64) -> int32 [L][k]."""
    s = np.ascontiguousarray(np.atleast_2d(np.asarray(sigma, dtype=np.float64)))
    L, T = s.shape
    if not 0 <= k <= T:
        raise ValueError("k outside [0, T]")
    out = np.zeros((L, k), dtype=np.int32)
    _load().oracle_select_hd(_ptr(s), L, T, int(k), _ptr(out))
    return out


def gather_kv_retained(ref_k, ref_v, idx, retained, cap: int | None = None, out_k=None, out_v=None):
    """Retention-aware rearrangement (Sec. 3.3.4, App. A): ref_k/ref_v [L][H][N][hd] (one
    reference prompt), idx [n_tgt], retained: L sequences of target tokens (layer l keeps
    retained[l]).  out[l][h][r] = ref[l][h][idx[retained[l][r]]], out [L][H][cap][hd] (cap
    defaults to the longest list; other rows stay as given, zeros when allocated here).
    Returns (out_k, out_v, n_bad)."""
    ref_k = np.ascontiguousarray(ref_k)
    ref_v = np.ascontiguousarray(ref_v)
    L, H, N, hd = ref_k.shape
    idx = np.ascontiguousarray(np.asarray(idx, dtype=np.int32))
    if len(retained) != L:
        raise ValueError("one retained list per layer")
    off = np.zeros(L + 1, dtype=np.int64)
    for l, r in enumerate(retained):
        off[l + 1] = off[l] + len(r)
    flat = np.ascontiguousarray(np.concatenate([np.asarray(r, dtype=np.int32) for r in retained])
                                if off[-1] else np.zeros(1, dtype=np.int32))
    cap = int(max((len(r) for r in retained), default=0)) if cap is None else int(cap)
    if out_k is None:
        out_k = np.zeros((L, H, cap, hd), dtype=ref_k.dtype)
    if out_v is None:
        out_v = np.zeros((L, H, cap, hd), dtype=ref_v.dtype)
    bad = _load().oracle_gather_kv_retained(_ptr(ref_k), _ptr(ref_v), L, H, N, hd * ref_k.dtype.itemsize, _ptr(idx),
                                            len(idx), _ptr(flat), _ptr(off), cap, _ptr(out_k), _ptr(out_v))
    return out_k, out_v, int(bad)


def fetch_rows(seg_k, seg_v, idx, dev_k=None, dev_v=None):
    """Selected-row load (Sec. 3.2, Sec. 3.3): seg_k/seg_v one [L][H][n_s][hd] array per reference
    segment (or a single array); dev_k/dev_v arrays of the same shapes (zeros when None) receive,
    for every l, h, the rows named in idx (global rows, any order, repeats allowed); all other
    rows stay as given.  Returns (dev_k, dev_v, n_bad), lists when seg_k is a list."""
    as_list = not isinstance(seg_k, np.ndarray)
    seg_k = [np.ascontiguousarray(a) for a in (seg_k if as_list else [seg_k])]
    seg_v = [np.ascontiguousarray(a) for a in (seg_v if as_list else [seg_v])]
    L, H, _, hd = seg_k[0].shape
    dt = seg_k[0].dtype
    if dev_k is None:
        dev_k = [np.zeros_like(a) for a in seg_k]
    if dev_v is None:
        dev_v = [np.zeros_like(a) for a in seg_v]
    dev_k = [dev_k] if isinstance(dev_k, np.ndarray) else list(dev_k)
    dev_v = [dev_v] if isinstance(dev_v, np.ndarray) else list(dev_v)
    offs = np.zeros(len(seg_k) + 1, dtype=np.int64)
    for s, a in enumerate(seg_k):
        if a.shape[:2] != (L, H) or a.shape[3] != hd or seg_v[s].shape != a.shape:
            raise ValueError("segment shapes differ")
        if dev_k[s].shape != a.shape or dev_v[s].shape != a.shape or not dev_k[s].flags.c_contiguous \
                or not dev_v[s].flags.c_contiguous:
            raise ValueError("dev arrays must be contiguous and shaped like the segments")
        offs[s + 1] = offs[s] + a.shape[2]
    idx = np.ascontiguousarray(np.asarray(idx, dtype=np.int32).ravel())
    n = len(seg_k)
    arr = lambda xs: (ctypes.c_void_p * n)(*[a.ctypes.data for a in xs])  # noqa: E731
    bad = _load().oracle_fetch_rows(arr(seg_k), arr(seg_v), arr(dev_k), arr(dev_v), _ptr(offs), n, L, H,
                                    hd * dt.itemsize, _ptr(idx), len(idx))
    return (dev_k, dev_v, int(bad)) if as_list else (dev_k[0], dev_v[0], int(bad))

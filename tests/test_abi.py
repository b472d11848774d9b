"""The C-ABI library loads, exports every declared entry point and rejects bad arguments on the
host, before touching the GPU (these tests run without one)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2509_24832_gb300 import build

    build.build()
    import paper_2509_24832_gb300 as ss

    return ss.load()


@pytest.fixture(scope="module")
def probe_lib(lib):
    from paper_2509_24832_gb300 import build

    p = ctypes.CDLL(build.PROBE_LIB)
    p.semshare_probe_hamming_rate.argtypes = [ctypes.c_int64, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]
    return p


@pytest.fixture(scope="module")
def checked_lib(lib):
    from paper_2509_24832_gb300 import build

    c = ctypes.CDLL(build.CHECKED_LIB)
    c.semshare_check_selftest.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    return c


def test_checked_build_exports_the_same_entry_points(lib, checked_lib):
    """libsemshare_checked.so: the same library with the bookkeeping checks compiled in."""
    for n in _declared("semshare.h"):
        assert hasattr(checked_lib, n), n
    assert lib.semshare_checked_build() == 0 and checked_lib.semshare_checked_build() == 1
    assert lib.semshare_check_selftest(None, None) == 2              # EUNSUPPORTED: plain build
    assert checked_lib.semshare_check_selftest(None, None) == 1      # EINVAL: no error word


def _declared(header):
    text = open(os.path.join(ROOT, "include", header)).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(semshare_\w+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib, probe_lib):
    assert sorted(f for f in os.listdir(os.path.join(ROOT, "include")) if f.endswith(".h")) == \
        ["semshare.h", "semshare_probe.h"]
    names = _declared("semshare.h")
    assert {"semshare_hash", "semshare_match", "semshare_gather_kv", "semshare_rope_table"} <= set(names)
    for n in names:
        assert hasattr(lib, n), n
    probes = _declared("semshare_probe.h")
    assert probes == ["semshare_probe_hamming_rate", "semshare_probe_hamming_threads"]
    for n in probes:
        assert hasattr(probe_lib, n), n
        assert not hasattr(lib, n), f"{n} is measurement support: it belongs to libsemshare_probe.so only"


def test_headers_are_plain_c_and_every_declaration_links(lib, probe_lib, tmp_path):
    """A C99 program that includes both headers and takes the address of every declared entry
    point compiles warning-free with -pedantic and links against the two libraries: the C ABI is
    plain C (no C++ types leak into it) and each declaration resolves to an exported symbol."""
    import shutil
    import subprocess

    from paper_2509_24832_gb300 import build

    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    names = _declared("semshare.h") + _declared("semshare_probe.h")
    src = tmp_path / "abi.c"
    src.write_text('#include "semshare.h"\n#include "semshare_probe.h"\n#include <stdio.h>\n'
                   "int main(void) {\n    void (*volatile p)(void) = 0;\n"
                   + "".join(f"    p = (void (*)(void)){n}; printf(\"%p\\n\", (void*)p);\n" for n in names)
                   + "    return 0;\n}\n")
    libdir = os.path.dirname(build.LIB)
    out = tmp_path / "abi"
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-Wno-pedantic",
                        "-I", os.path.join(ROOT, "include"), str(src), "-o", str(out), "-L", libdir,
                        "-lsemshare", "-lsemshare_probe", f"-Wl,-rpath,{libdir}"],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-fsyntax-only",
                        "-I", os.path.join(ROOT, "include"), "-x", "c", "-"],
                       input='#include "semshare.h"\n#include "semshare_probe.h"\n', capture_output=True, text=True)
    assert r.returncode == 0 and not r.stderr.strip(), r.stderr


def test_status_helpers(lib):
    assert lib.semshare_abi_version() == 1
    assert lib.semshare_status_string(0) == b"ok"
    assert lib.semshare_flag_status(0) == 0
    assert lib.semshare_flag_status(1) == 4
    assert lib.semshare_flag_status(3) == 5
    assert lib.semshare_flag_status(4) == 7                        # a failed check (checked build)
    assert lib.semshare_flag_status(5 | (3 << 8) | (123 << 16)) == 7
    assert lib.semshare_flag_status(6) == 5                        # a timeout wins
    assert lib.semshare_status_string(7).startswith(b"checked build")
    assert lib.semshare_match_workspace_size(1000) == 8000


FAKE = ctypes.c_void_p(1 << 20)  # aligned, never dereferenced: every case below fails validation first


def _hash(lib, **kw):
    a = dict(emb=FAKE, dtype=0, n=10, d=128, row_stride=128, positions=None, table=FAKE, hyp=FAKE, nbits=64,
             codes=FAKE, proj=None, ws=FAKE, ws_bytes=1 << 30, flag=None, stream=None)
    a.update(kw)
    return lib.semshare_hash(a["emb"], a["dtype"], a["n"], a["d"], a["row_stride"], a["positions"], a["table"],
                             a["hyp"], a["nbits"], a["codes"], a["proj"], a["ws"], a["ws_bytes"], a["flag"],
                             a["stream"])


def test_hash_argument_errors(lib):
    assert _hash(lib, dtype=7) == 1
    assert _hash(lib, n=-1) == 1
    assert _hash(lib, d=127, row_stride=127) == 1
    assert _hash(lib, d=96, row_stride=96) == 2          # d not a multiple of 64
    assert _hash(lib, nbits=48) == 2
    assert _hash(lib, nbits=288) == 2
    assert _hash(lib, row_stride=100) == 1               # shorter than d
    assert _hash(lib, row_stride=132) == 1               # 264-byte rows: not 16-byte multiple
    assert _hash(lib, emb=None) == 1
    assert _hash(lib, emb=ctypes.c_void_p((1 << 20) + 4)) == 1  # misaligned
    assert _hash(lib, codes=None) == 1
    assert _hash(lib, n=1 << 31) == 2
    assert _hash(lib, ws=None) == 1
    assert _hash(lib, ws=ctypes.c_void_p((1 << 20) + 16)) == 1  # workspace not 256-byte aligned
    assert _hash(lib, n=0, emb=None, codes=None) == 0    # empty: nothing to do


def test_hash_ex_argument_errors(lib):
    def hx(layout, dtype=0, d=128):
        return lib.semshare_hash_ex(FAKE, dtype, 10, d, d, None, FAKE, FAKE, 64, layout, FAKE, None, FAKE, 1 << 30,
                                    None, None)
    assert hx(3) == 1                    # unknown pairing
    # no rotation (2) needs no rotation table: the call gets past the table check and stops at the
    # device query (no GPU: ECUDA) or at the empty workspace (EINVAL) -- nothing is launched;
    # with a rotation a missing table is an argument error
    nt = lib.semshare_hash_ex(FAKE, 0, 10, 128, 128, None, None, FAKE, 64, 2, FAKE, None, FAKE, 0, None, None)
    assert nt in (1, 3)
    assert lib.semshare_hash_ex(FAKE, 0, 10, 128, 128, None, None, FAKE, 64, 0, FAKE, None, FAKE, 1 << 30, None,
                                None) == 1
    assert hx(1, dtype=1) == 2           # rotate-half takes bf16 rows
    assert hx(1, d=192) == 2             # and d a multiple of 128
    assert lib.semshare_hash_ex(None, 0, 0, 128, 128, None, None, None, 64, 1, None, None, None, 0, None,
                                None) == 0  # empty


def test_hash_pair_argument_errors(lib):
    hp = lib.semshare_hash_pair
    assert hp(FAKE, 0, 10, 128, 128, None, FAKE, FAKE, 64, FAKE, None, FAKE, 1 << 30, None, None) == 1  # no 2nd output
    assert hp(FAKE, 0, 1 << 30, 128, 128, None, FAKE, FAKE, 64, FAKE, FAKE, FAKE, 1 << 30, None, None) == 2  # too many
    odd = ctypes.c_void_p((1 << 20) + 4)
    assert hp(FAKE, 0, 10, 128, 128, None, FAKE, FAKE, 64, FAKE, odd, FAKE, 1 << 30, None, None) in (1, 3)
    assert hp(None, 0, 0, 128, 128, None, None, None, 64, None, None, None, 0, None, None) == 0  # empty
    assert lib.semshare_hash_pair_workspace_size(0, 128, 64) == 0


def test_hash_signs_argument_errors(lib):
    hs = lib.semshare_hash_signs
    odd = ctypes.c_void_p((1 << 20) + 8)

    def call(signs=FAKE, n=10, layout=0, codes2_like=None):
        return hs(FAKE, 0, n, 128, 128, None, FAKE, FAKE, 64, layout, FAKE, signs, None, FAKE, 1 << 30, None, None)

    assert call(signs=None) == 1                       # the sign rows are the point of the call
    assert call(signs=odd) == 1                        # not 16-byte aligned
    assert call(layout=3) == 1
    assert call(n=0, signs=None) == 0                  # empty
    assert [lib.semshare_signs_pitch(b) for b in (32, 64, 96, 128, 160, 256)] == [128, 128, 128, 128, 256, 256]
    assert lib.semshare_signs_pitch(48) == 0 and lib.semshare_signs_pitch(288) == 0


def test_match_tc_signs_argument_errors(lib):
    m = lib.semshare_match_tc_signs
    odd = ctypes.c_void_p((1 << 20) + 8)
    ws = lib.semshare_match_tc_signs_workspace_size(10)
    assert ws == 256 + 256                              # 10 keys rounded to 256 bytes, then the counter
    assert lib.semshare_match_tc_signs_workspace_size(0) == 0
    assert m(FAKE, 10, FAKE, 0, 64, FAKE, None, FAKE, ws, None, None) == 1      # n_ref = 0
    assert m(FAKE, 10, FAKE, 5, 40, FAKE, None, FAKE, ws, None, None) == 2      # nbits
    assert m(FAKE, 10, FAKE, 5, 64, FAKE, None, FAKE, ws - 1, None, None) == 1  # workspace too small
    assert m(odd, 10, FAKE, 5, 64, FAKE, None, FAKE, ws, None, None) == 1       # TMA rows: 16-byte aligned
    assert m(FAKE, 10, FAKE, 5, 64, None, None, FAKE, ws, None, None) == 1
    assert m(None, 0, FAKE, 5, 64, None, None, None, 0, None, None) == 0        # empty target


def test_match_argument_errors(lib):
    m = lib.semshare_match
    assert m(FAKE, 10, FAKE, 0, 64, FAKE, None, FAKE, 80, None) == 1   # n_ref = 0
    assert m(FAKE, 10, FAKE, 5, 40, FAKE, None, FAKE, 80, None) == 2   # nbits
    assert m(FAKE, 10, FAKE, 5, 64, FAKE, None, FAKE, 79, None) == 1   # workspace too small
    assert m(FAKE, 10, FAKE, 5, 64, None, None, FAKE, 80, None) == 1
    assert m(None, 0, FAKE, 5, 64, None, None, None, 0, None) == 0     # empty target


def test_gather_argument_errors(lib):
    import paper_2509_24832_gb300 as ss

    lay = ss.KVLayout(2, 4, 64, 2, 0, 4 * 100 * 64, 100 * 64, 64)
    out = ss.KVLayout(2, 4, 64, 2, 2 * 4 * 10 * 64, 4 * 10 * 64, 10 * 64, 64)
    pk = (ctypes.c_void_p * 1)(1 << 20)
    offs = (ctypes.c_int64 * 2)(0, 100)
    g = lib.semshare_gather_kv
    assert g(pk, pk, offs, 0, lay, FAKE, 10, 1, FAKE, FAKE, out, None, None) == 1       # n_seg
    bad = ss.KVLayout(2, 4, 60, 2, 0, 4 * 100 * 60, 100 * 60, 60)                        # 120-byte rows
    assert g(pk, pk, offs, 1, bad, FAKE, 10, 1, FAKE, FAKE, bad, None, None) == 1
    other = ss.KVLayout(2, 8, 64, 2, 0, 8 * 100 * 64, 100 * 64, 64)
    assert g(pk, pk, offs, 1, lay, FAKE, 10, 1, FAKE, FAKE, other, None, None) == 1     # head mismatch
    offs_bad = (ctypes.c_int64 * 2)(5, 100)
    assert g(pk, pk, offs_bad, 1, lay, FAKE, 10, 1, FAKE, FAKE, out, None, None) == 1
    assert g(pk, pk, offs, 1, lay, None, 0, 1, None, None, out, None, None) == 0        # empty


def test_retrieve_argument_errors(lib):
    r = lib.semshare_retrieve

    def call(offs, n_cand=None, n_tgt=10, nbits=64, max_dist=30.0, thr=0.8, best=FAKE, ws_bytes=1 << 30):
        o = (ctypes.c_int64 * len(offs))(*offs)
        n_cand = len(offs) - 1 if n_cand is None else n_cand
        return r(FAKE, n_tgt, FAKE, o, n_cand, nbits, max_dist, thr, None, None, best, None, None, None, FAKE,
                 ws_bytes, None, None)

    assert call([0]) == 1                              # no candidate
    assert call([0, 5, 5, 9]) == 1                     # empty candidate
    assert call([1, 5]) == 1                           # does not start at row 0
    assert call([0, 5, 3]) == 1                        # decreasing
    assert call(list(range(258))) == 2                 # 257 candidates: above the maximum
    assert call([0, 5], nbits=40) == 2
    assert call([0, 5], n_tgt=0) == 1                  # the mean over no target token
    assert call([0, 5], max_dist=0.0) == 1
    assert call([0, 5], thr=float("nan")) == 1
    assert call([0, 5], best=None) == 1
    assert call([0, 5], ws_bytes=100) == 1             # workspace too small
    assert lib.semshare_retrieve_workspace_size(10, 5, 0, 64) == 0
    assert lib.semshare_retrieve_workspace_size(10, 5, 1, 64) > lib.semshare_match_tc_workspace_size(10, 5, 64)


def test_match_selected_argument_errors(lib):
    m = lib.semshare_match_tc_selected

    def call(offs, n_tgt=10, nbits=64, best=FAKE, ws_bytes=1 << 30, n_cand=None):
        o = (ctypes.c_int64 * len(offs))(*offs)
        n_cand = len(offs) - 1 if n_cand is None else n_cand
        return m(FAKE, n_tgt, FAKE, o, n_cand, best, nbits, FAKE, None, FAKE, ws_bytes, None, None)

    assert call([0, 5, 5]) == 1                        # empty candidate
    assert call([1, 5]) == 1                           # does not start at row 0
    assert call(list(range(258))) == 2                 # 257 candidates
    assert call([0, 5], nbits=40) == 2
    assert call([0, 5], best=None) == 1
    assert call([0, 5], ws_bytes=100) == 1
    assert call([0, 5], n_tgt=0) == 0                  # nothing to match
    o = (ctypes.c_int64 * 3)(0, 300, 400)
    assert lib.semshare_match_tc_selected_workspace_size(10, o, 2, 64) == \
        lib.semshare_match_tc_workspace_size(10, 300, 64) + 256     # sized for the longest candidate


def test_gather_retained_argument_errors(lib):
    import paper_2509_24832_gb300 as ss

    lay = ss.KVLayout(2, 4, 64, 2, 0, 4 * 100 * 64, 100 * 64, 64)
    out = ss.KVLayout(2, 4, 64, 2, 0, 4 * 10 * 64, 10 * 64, 64)
    pk = (ctypes.c_void_p * 1)(1 << 20)
    offs = (ctypes.c_int64 * 2)(0, 100)
    g = lib.semshare_gather_kv_retained

    def ro(*v):
        return (ctypes.c_int64 * len(v))(*v)

    assert g(pk, pk, offs, 1, lay, FAKE, 10, FAKE, None, FAKE, FAKE, out, None, None) == 1        # no offsets
    assert g(pk, pk, offs, 1, lay, FAKE, 10, FAKE, ro(1, 5, 9), FAKE, FAKE, out, None, None) == 1  # not from 0
    assert g(pk, pk, offs, 1, lay, FAKE, 10, FAKE, ro(0, 5, 3), FAKE, FAKE, out, None, None) == 1  # decreasing
    assert g(pk, pk, offs, 1, lay, None, 10, FAKE, ro(0, 5, 9), FAKE, FAKE, out, None, None) == 1  # no idx
    deep = ss.KVLayout(129, 4, 64, 2, 0, 4 * 100 * 64, 100 * 64, 64)
    assert g(pk, pk, offs, 1, deep, FAKE, 10, FAKE, ro(*([0] * 130)), FAKE, FAKE, deep, None, None) == 2
    assert g(pk, pk, offs, 1, lay, None, 10, None, ro(0, 0, 0), None, None, out, None, None) == 0  # nothing kept


def test_fetch_argument_errors(lib):
    import paper_2509_24832_gb300 as ss

    lay = ss.KVLayout(2, 4, 64, 2, 0, 4 * 100 * 64, 100 * 64, 64)
    pk = (ctypes.c_void_p * 1)(1 << 20)
    pd = (ctypes.c_void_p * 1)(1 << 21)
    offs = (ctypes.c_int64 * 2)(0, 100)
    f = lib.semshare_fetch_rows
    ws = lib.semshare_fetch_workspace_size(100)
    assert ws >= 100 and lib.semshare_fetch_workspace_size(0) == 0
    assert f(pk, pk, pd, pd, offs, 0, lay, FAKE, 10, FAKE, ws, None, None) == 1            # n_seg
    bad = ss.KVLayout(2, 4, 60, 2, 0, 4 * 100 * 60, 100 * 60, 60)                           # 120-byte rows
    assert f(pk, pk, pd, pd, offs, 1, bad, FAKE, 10, FAKE, ws, None, None) == 1
    odd = ss.KVLayout(2, 4, 64, 2, 0, 4 * 100 * 64 + 4, 100 * 64, 64)                       # stride not 16 B
    assert f(pk, pk, pd, pd, offs, 1, odd, FAKE, 10, FAKE, ws, None, None) == 1
    nul = (ctypes.c_void_p * 1)(None)
    assert f(pk, pk, nul, pd, offs, 1, lay, FAKE, 10, FAKE, ws, None, None) == 1            # no destination
    assert f(pk, pk, pd, pd, offs, 1, lay, None, 10, FAKE, ws, None, None) == 1             # no idx
    assert f(pk, pk, pd, pd, offs, 1, lay, FAKE, 10, FAKE, ws - 1, None, None) == 1        # workspace too small
    assert f(pk, pk, pd, pd, offs, 1, lay, FAKE, -1, FAKE, ws, None, None) == 1             # negative count
    offs_bad = (ctypes.c_int64 * 2)(5, 100)
    assert f(pk, pk, pd, pd, offs_bad, 1, lay, FAKE, 10, FAKE, ws, None, None) == 1
    huge = (ctypes.c_int64 * 2)(0, 1 << 31)
    assert f(pk, pk, pd, pd, huge, 1, lay, FAKE, 10, FAKE, ws, None, None) == 2
    assert f(pk, pk, pd, pd, offs, 1, lay, None, 0, None, 0, None, None) == 0               # empty


def test_probe_argument_errors(probe_lib):
    p = probe_lib.semshare_probe_hamming_rate
    assert p(0, FAKE, 1 << 30, None) == 1               # no iterations
    assert p((1 << 24) + 1, FAKE, 1 << 30, None) == 1   # too many
    assert p(16, None, 1 << 30, None) == 1              # no sink


def test_deviation_and_select_argument_errors(lib):
    import paper_2509_24832_gb300 as ss

    lay = ss.KVLayout(1, 8, 128, 2, 0, 8 * 100 * 128, 100 * 128, 128)
    d = lib.semshare_kv_deviation
    assert d(FAKE, FAKE, lay, FAKE, FAKE, lay, 7, 100, None, None, FAKE, None) == 1       # dtype
    assert d(FAKE, FAKE, lay, FAKE, FAKE, lay, 1, 100, None, None, FAKE, None) == 1       # f32 vs 2-byte elements
    other = ss.KVLayout(1, 4, 128, 2, 0, 4 * 100 * 128, 100 * 128, 128)
    assert d(FAKE, FAKE, lay, FAKE, FAKE, other, 0, 100, None, None, FAKE, None) == 1     # head mismatch
    odd = ss.KVLayout(1, 8, 60, 2, 0, 8 * 100 * 60, 100 * 60, 60)                         # 120-byte rows
    assert d(FAKE, FAKE, odd, FAKE, FAKE, odd, 0, 100, None, None, FAKE, None) == 1
    assert d(FAKE, FAKE, lay, FAKE, FAKE, lay, 0, 100, None, None, None, None) == 1       # no sigma_kv
    assert d(ctypes.c_void_p((1 << 20) + 8), FAKE, lay, FAKE, FAKE, lay, 0, 100, None, None, FAKE, None) == 1
    assert d(None, None, lay, None, None, lay, 0, 0, None, None, None, None) == 0         # empty
    s = lib.semshare_select_hd
    assert s(FAKE, 1, 100, 101, FAKE, None, None) == 1                                    # k > n_tok
    assert s(FAKE, 1, 100, -1, FAKE, None, None) == 1
    assert s(FAKE, 1, 100, 10, None, None, None) == 1                                     # no output
    assert s(FAKE, 70000, 100, 10, FAKE, None, None) == 2                                 # too many layers
    assert s(None, 1, 0, 0, None, None, None) == 0                                        # empty


def test_rope_table_argument_errors(lib):
    t = lib.semshare_rope_table
    assert t(7, 10000.0, FAKE, None) == 1
    assert t(64, 0.0, FAKE, None) == 1
    assert t(64, float('nan'), FAKE, None) == 1
    assert t(64, 10000.0, None, None) == 1


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    import paper_2509_24832_gb300._native as nat

    monkeypatch.setattr(nat, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(nat, "_lib", None)
    with pytest.raises(RuntimeError):
        nat.load()

"""The C-ABI library builds, loads and exports every entry point that
include/presto.h declares; host-side validation rejects bad arguments before any
work is enqueued.  No kernel runs here (CPU only)."""

import ctypes
import os
import re

import pytest

import paper_2607_22634_gb300 as P
from paper_2607_22634_gb300 import _lib

HDR = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "presto.h")


def declared_functions():
    src = open(HDR).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b(presto_\w+)\s*\(", src, flags=re.M)
    inline = set(re.findall(r"static\s+inline\s+\w+\s+(presto_\w+)", src))
    return sorted(set(names) - inline)


def test_header_declares_the_five_steps():
    names = declared_functions()
    for n in ("presto_topk", "presto_score_build_tree", "presto_tree_mask",
              "presto_tree_attention", "presto_accept"):
        assert n in names


def test_library_exports_every_declared_symbol():
    lib = ctypes.CDLL(P.load() and _lib.lib_path())
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing
    # and the binding declares a signature for each of them
    assert set(declared_functions()) <= set(_lib._SIGS)


def test_version_and_status_strings():
    lib = P.load()
    assert lib.presto_version() >> 16 == 1
    for code in (0, -1, -2, -3, -4):
        assert lib.presto_status_string(code).startswith(b"PRESTO")


N = None


def test_host_validation_rejects_bad_arguments():
    lib = P.load()
    p = ctypes.c_void_p(16)  # never dereferenced: every call below fails validation first
    # null logits
    assert lib.presto_topk(N, 1, 1, 1, 10, 10, 2, p, p, N, N, 0, N, N) == -1
    # bad dtype
    assert lib.presto_topk(p, 7, 1, 1, 10, 10, 2, p, p, N, N, 0, N, N) == -1
    # k > V
    assert lib.presto_topk(p, 1, 1, 1, 4, 4, 5, p, p, N, N, 0, N, N) == -1
    # k above the packing limit
    assert lib.presto_topk(p, 1, 1, 1, 100, 100, 17, p, p, N, N, 0, N, N) == -2
    # V beyond 2^18
    assert lib.presto_topk(p, 1, 1, 1, 1 << 18, 1 << 18, 4, p, p, N, N, 0, N, N) == -2
    # row stride below V
    assert lib.presto_topk(p, 1, 1, 1, 100, 99, 4, p, p, N, N, 0, N, N) == -1
    # build: b > k, N > 1024, negative lambda
    args = lambda B, L, k, b, lam, Nn: (p, p, B, L, k, b, p, None, ctypes.c_float(lam), Nn,
                                        p, p, p, p, p, N, 0, N, N)
    assert lib.presto_score_build_tree(*args(1, 4, 4, 5, 0.2, 8)) == -1
    assert lib.presto_score_build_tree(*args(1, 4, 4, 4, 0.2, 1025)) == -2
    assert lib.presto_score_build_tree(*args(1, 4, 4, 4, -0.5, 8)) == -1
    assert lib.presto_score_build_tree(*args(1, 64, 4, 4, 0.2, 8)) == -2
    # build_ex: unknown policy, beam width 0 or above 1024
    ex = lambda pol, W: (p, p, 1, 4, 4, 4, p, None, ctypes.c_float(0.2), N, pol, W, 8,
                         p, p, p, p, p, N, 0, N, N)
    assert lib.presto_score_build_tree_ex(*ex(3, 1)) == -1
    assert lib.presto_score_build_tree_ex(*ex(1, 0)) == -1
    assert lib.presto_score_build_tree_ex(*ex(1, 1025)) == -2
    # build_tree_mask: kv_len, mask and pos_ids come together
    bm = lambda kv, mk, po: (p, p, 1, 4, 4, 4, p, None, ctypes.c_float(0.2), N, 0, 1, 8,
                             p, p, p, p, p, kv, mk, po, N, 0, N, N)
    assert lib.presto_score_build_tree_mask(*bm(p, N, p)) == -1
    assert lib.presto_score_build_tree_mask(*bm(N, p, N)) == -1
    # topk_entropy: no output, beta or C not positive and finite
    f = ctypes.c_float
    ent = lambda beta, c, H, lam: (p, 1, 1, 1, 10, 10, 2, f(beta), f(c), p, p, N, H, lam, N, 0,
                                   N, N)
    assert lib.presto_topk_entropy(*ent(1.0, 1.0, N, N)) == -1
    assert lib.presto_topk_entropy(*ent(0.0, 1.0, N, p)) == -1
    assert lib.presto_topk_entropy(*ent(1.0, -1.0, N, p)) == -1
    assert lib.presto_topk_entropy(*ent(1.0, float("inf"), p, p)) == -1
    assert lib.presto_topk_entropy(*ent(1.0, float("nan"), N, p)) == -1
    # mask: N beyond limit
    assert lib.presto_tree_mask(p, p, p, p, 1, 1100, p, p, N, N) == -2
    # attention: head dim, GQA ratio, misalignment
    att = lambda D, Hq, Hkv, q=p: (q, p, p, p, 64, p, p, p, p, 1, 8, Hq, Hkv, D,
                                   ctypes.c_float(0.1), p, N, N, 0, N, N)
    assert lib.presto_tree_attention(*att(96, 8, 2)) == -2
    assert lib.presto_tree_attention(*att(128, 12, 4)) == -2      # G = 3 not a power of two
    assert lib.presto_tree_attention(*att(128, 8, 3)) == -1       # Hq % Hkv != 0
    assert lib.presto_tree_attention(*att(128, 8, 2, q=ctypes.c_void_p(24))) == -1
    # attention queries: refused shapes size nothing and launch nothing (answered on the
    # host, before any CUDA call)
    for B, Nn, Hq, Hkv, D, T in ((0, 8, 8, 2, 128, 64), (1, 8, 8, 3, 128, 64),
                                 (1, 8, 8, 2, 96, 64), (1, 8, 8, 2, 128, 0)):
        assert lib.presto_attn_workspace(B, Nn, Hq, Hkv, D, T) == 0
        assert lib.presto_attn_launches(B, Nn, Hq, Hkv, D, T) == 0
    # accept: L above limit
    assert lib.presto_accept(p, p, p, p, p, p, 1, 8, 64, p, p, p, N, N) == -2
    # table: capacity out of range
    bad = _lib.Ngram3(16, 16, 40, -12.0)
    assert lib.presto_ngram3_clear(ctypes.byref(bad), N) == -1
    # wait self-test: a status word is required; the limit stays within the library's
    assert lib.presto_selftest_wait_timeout(N, 1000, N) == -1
    assert lib.presto_selftest_wait_timeout(p, -1, N) == -1
    assert lib.presto_selftest_wait_timeout(p, 3_000_000_000, N) == -1


def test_binding_raises_on_error_status():
    with pytest.raises(_lib.PrestoError):
        _lib._check(-2, "x")


def test_trigram_key_packing():
    k = _lib.pack_trigram_keys([1, 262143], [2, 0], [3, 262143])
    assert int(k[0]) == (1 << 36) | (2 << 18) | 3
    assert int(k[1]) == (262143 << 36) | 262143


def test_noalloc_build_host_checks():
    """presto_score_build_tree_noalloc refuses, on the host and before any CUDA call,
    shapes whose scratch exceeds its fixed 1 MiB array and malformed shapes; the
    workspace query agrees on which shapes need more than the array holds."""
    lib = P.load()
    p = ctypes.c_void_p(16)  # never dereferenced: every call below is refused first
    call = lambda B, L, k, b, Nn, W=1, lam=0.2, tbl=None: lib.presto_score_build_tree_noalloc(
        p, p, B, L, k, b, p, tbl, ctypes.c_float(lam), N, 0 if W == 1 else 1, W, Nn,
        p, p, p, p, p, N, N, N, N, N)
    desc = ctypes.byref(_lib.Ngram3(16, 16, 20, -12.0))
    # three N = 1024 trees (k = b = 8, with a table): ~1.18 MB of selection scratch
    assert lib.presto_build_workspace_ex(3, 16, 8, 1024, 1) > (1 << 20)
    assert call(3, 16, 8, 8, 1024, tbl=desc) == -2
    # malformed shapes and limits
    assert call(0, 16, 8, 8, 64) == -1
    assert call(1, 16, 8, 9, 64) == -1        # b > k
    assert call(1, 64, 8, 8, 64) == -2        # L above the limit
    assert call(1, 16, 17, 8, 64) == -2       # k above the limit
    assert call(1, 16, 8, 8, 1025) == -2      # N above the limit
    assert call(1, 16, 8, 8, 64, W=0) == -1   # beam width 0
    # pointer, lambda, policy and table checks also run before the scratch lookup:
    # here, with no GPU at all, each call still returns INVALID_ARG rather than a CUDA
    # error
    f = ctypes.c_float
    full = lambda ids=p, lam=0.2, pol=0, tbl=None, kv=N, mk=N, po=N: \
        lib.presto_score_build_tree_noalloc(ids, p, 1, 16, 8, 8, p, tbl, f(lam), N, pol, 1, 64,
                                            p, p, p, p, p, kv, mk, po, N, N)
    assert full(ids=N) == -1                  # null candidate ids
    assert full(lam=-0.5) == -1               # negative lambda
    assert full(lam=float("nan")) == -1
    assert full(pol=3) == -1                  # unknown search policy
    assert full(tbl=ctypes.byref(_lib.Ngram3(16, 16, 40, -12.0))) == -1  # table capacity
    assert full(tbl=ctypes.byref(_lib.Ngram3(16, 16, 20, 0.5))) == -1    # miss log rho > 0
    assert full(kv=p) == -1                   # kv_len without mask and pos_ids

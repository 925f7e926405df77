"""ctypes binding to libpresto.so: the C-ABI entry points under the same names.

Argument marshalling only.  Tensors are passed by device pointer on the current
torch stream; outputs and workspaces the caller does not pass are allocated with
torch (device memory is PyTorch's job here).  Every step of the computation runs
in the library's CUDA kernels; if the library cannot be loaded, every call raises.
"""

from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

from . import build as _build

_HERE = os.path.dirname(os.path.abspath(__file__))

PRESTO_OK = 0
PRESTO_F32 = 0
PRESTO_BF16 = 1
NGRAM3_EMPTY = 0xFFFFFFFFFFFFFFFF

DEV_STATUS_BITS = {
    0x1: "BAD_PARENT", 0x2: "BAD_TOKEN", 0x4: "BAD_KVLEN", 0x8: "BAD_NNODES",
    0x10: "POSITIVE_SCORE", 0x20: "TIMEOUT", 0x40: "DUP_SIBLING", 0x80: "TABLE_FULL",
    0x100: "NONFINITE", 0x200: "BAD_PATH", 0x400: "BOUNDS",
}
BUILD_CHECKS = 0x1  # presto_build_flags(): compiled with device-side bounds checks


class Ngram3(ctypes.Structure):
    _fields_ = [("keys", ctypes.c_void_p), ("logrho", ctypes.c_void_p),
                ("log2_cap", ctypes.c_uint32), ("miss_logrho", ctypes.c_float)]


class PrestoError(RuntimeError):
    pass


_P = ctypes.c_void_p
_I = ctypes.c_int
_SIGS = {
    "presto_status_string": (ctypes.c_char_p, [_I]),
    "presto_version": (_I, []),
    "presto_topk_workspace": (ctypes.c_size_t, [_I, _I, _I, _I]),
    "presto_topk": (_I, [_P, _I, _I, _I, _I, ctypes.c_longlong, _I, _P, _P, _P, _P,
                         ctypes.c_size_t, _P, _P]),
    "presto_topk_slots": (_I, [_P, _I, _I, _I, _I, _I, ctypes.c_longlong, _P, _P, _I, _I, _I, _I,
                               _P, _P, _P, _P, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "presto_topk_entropy": (_I, [_P, _I, _I, _I, _I, ctypes.c_longlong, _I, ctypes.c_float,
                                 ctypes.c_float, _P, _P, _P, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "presto_ngram3_clear": (_I, [ctypes.POINTER(Ngram3), _P]),
    "presto_ngram3_insert": (_I, [ctypes.POINTER(Ngram3), _P, _P, _I, _P, _P]),
    "presto_build_workspace": (ctypes.c_size_t, [_I, _I, _I, _I]),
    "presto_build_workspace_ex": (ctypes.c_size_t, [_I, _I, _I, _I, _I]),
    "presto_score_build_tree_ex": (_I, [_P, _P, _I, _I, _I, _I, _P, ctypes.POINTER(Ngram3),
                                        ctypes.c_float, _P, _I, _I, _I, _P, _P, _P, _P, _P,
                                        _P, ctypes.c_size_t, _P, _P]),
    "presto_score_build_tree_mask": (_I, [_P, _P, _I, _I, _I, _I, _P, ctypes.POINTER(Ngram3),
                                          ctypes.c_float, _P, _I, _I, _I, _P, _P, _P, _P, _P,
                                          _P, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "presto_score_build_tree_noalloc": (_I, [_P, _P, _I, _I, _I, _I, _P,
                                             ctypes.POINTER(Ngram3), ctypes.c_float, _P, _I, _I,
                                             _I, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P]),
    "presto_score_build_tree": (_I, [_P, _P, _I, _I, _I, _I, _P, ctypes.POINTER(Ngram3),
                                     ctypes.c_float, _I, _P, _P, _P, _P, _P, _P,
                                     ctypes.c_size_t, _P, _P]),
    "presto_tree_mask": (_I, [_P, _P, _P, _P, _I, _I, _P, _P, _P, _P]),
    "presto_attn_workspace": (ctypes.c_size_t, [_I, _I, _I, _I, _I, _I]),
    "presto_attn_launches": (_I, [_I, _I, _I, _I, _I, _I]),
    "presto_tree_attention": (_I, [_P, _P, _P, _P, _I, _P, _P, _P, _P, _I, _I, _I, _I, _I,
                                   ctypes.c_float, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "presto_accept": (_I, [_P, _P, _P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _P]),
    "presto_selftest_wait_timeout": (_I, [_P, ctypes.c_longlong, _P]),
    "presto_build_flags": (_I, []),
}

_lib = None


def lib_path() -> str:
    """The library this process loads (the bounds-checked debug build under
    PRESTO_CHECKS=1)."""
    return _build.lib_file()


def load(build_if_missing: bool = True):
    """Load the library (building it first if needed) and declare signatures."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.lib_file()
    if build_if_missing and not _build.up_to_date():
        _build.build()
    if not os.path.exists(path):
        raise PrestoError(f"{os.path.basename(path)} is missing; run paper_2607_22634_gb300.build.build()")
    lib = ctypes.CDLL(path)
    for name, (res, args) in _SIGS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _check(status: int, what: str):
    if status != PRESTO_OK:
        msg = load().presto_status_string(status).decode()
        raise PrestoError(f"{what}: {msg} ({status})")


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _need(t, dtype, shape, name):
    if t.dtype != dtype or tuple(t.shape) != tuple(shape) or not t.is_contiguous() or not t.is_cuda:
        raise ValueError(f"{name}: expected contiguous CUDA {dtype} {tuple(shape)}, "
                         f"got {t.dtype} {tuple(t.shape)} on {t.device}")
    return t


def _ws(nbytes, device, ws):
    if nbytes == 0:
        return None, 0
    if ws is None:
        ws = torch.empty(nbytes, dtype=torch.uint8, device=device)
    if ws.numel() < nbytes:
        raise ValueError(f"workspace too small: {ws.numel()} < {nbytes}")
    return ws, ws.numel()


def dev_status_names(code: int):
    return [n for bit, n in DEV_STATUS_BITS.items() if code & bit]


# ------------------------------------------------------------------ top-k

def presto_topk_workspace(B, L, V, k) -> int:
    return int(load().presto_topk_workspace(B, L, V, k))


def presto_topk(logits, k, topk_ids=None, topk_logq=None, lse=None, ws=None, dev_status=None,
                stream=None, with_lse=True):
    """logits [B, L, V'] (fp32 or bf16, last dim stride 1, V = V' unless sliced)."""
    if logits.dim() != 3 or logits.stride(2) != 1 or logits.stride(0) != logits.shape[1] * logits.stride(1):
        raise ValueError("logits must be [B, L, V] with unit last stride and packed rows")
    B, L, V = logits.shape
    dtype = {torch.float32: PRESTO_F32, torch.bfloat16: PRESTO_BF16}.get(logits.dtype)
    if dtype is None:
        raise ValueError("logits must be float32 or bfloat16")
    dev = logits.device
    topk_ids = torch.empty(B, L, k, dtype=torch.int32, device=dev) if topk_ids is None else topk_ids
    topk_logq = torch.empty(B, L, k, dtype=torch.float32, device=dev) if topk_logq is None else topk_logq
    if lse is None and with_lse:
        lse = torch.empty(B, L, dtype=torch.float32, device=dev)
    _need(topk_ids, torch.int32, (B, L, k), "topk_ids")
    _need(topk_logq, torch.float32, (B, L, k), "topk_logq")
    ws, nws = _ws(presto_topk_workspace(B, L, V, k), dev, ws)
    st = load().presto_topk(_ptr(logits), dtype, B, L, V, logits.stride(1), k, _ptr(topk_ids),
                            _ptr(topk_logq), _ptr(lse), _ptr(ws), nws, _ptr(dev_status),
                            _stream(stream))
    _check(st, "presto_topk")
    return topk_ids, topk_logq, lse


def presto_topk_entropy(logits, k, beta=None, C=None, topk_ids=None, topk_logq=None, lse=None,
                        entropy=None, lambda_d=None, ws=None, dev_status=None, stream=None,
                        with_lse=True, with_entropy=True, with_lambda=True):
    """presto_topk plus each row's entropy H_d and lambda_d = beta H_d / (H_d + C)
    (App. F).  Returns (topk_ids, topk_logq, lse, entropy, lambda_d); lambda_d is
    None unless beta and C are given."""
    if logits.dim() != 3 or logits.stride(2) != 1 or logits.stride(0) != logits.shape[1] * logits.stride(1):
        raise ValueError("logits must be [B, L, V] with unit last stride and packed rows")
    B, L, V = logits.shape
    dtype = {torch.float32: PRESTO_F32, torch.bfloat16: PRESTO_BF16}.get(logits.dtype)
    if dtype is None:
        raise ValueError("logits must be float32 or bfloat16")
    dev = logits.device
    f32 = torch.float32
    topk_ids = torch.empty(B, L, k, dtype=torch.int32, device=dev) if topk_ids is None else topk_ids
    topk_logq = torch.empty(B, L, k, dtype=f32, device=dev) if topk_logq is None else topk_logq
    if lse is None and with_lse:
        lse = torch.empty(B, L, dtype=f32, device=dev)
    if entropy is None and with_entropy:
        entropy = torch.empty(B, L, dtype=f32, device=dev)
    adaptive = beta is not None and C is not None
    if lambda_d is None and with_lambda and adaptive:
        lambda_d = torch.empty(B, L, dtype=f32, device=dev)
    _need(topk_ids, torch.int32, (B, L, k), "topk_ids")
    _need(topk_logq, f32, (B, L, k), "topk_logq")
    for t, name in ((lse, "lse"), (entropy, "entropy"), (lambda_d, "lambda_d")):
        if t is not None:
            _need(t, f32, (B, L), name)
    ws, nws = _ws(presto_topk_workspace(B, L, V, k), dev, ws)
    st = load().presto_topk_entropy(_ptr(logits), dtype, B, L, V, logits.stride(1), k,
                                    float(beta) if adaptive else 0.0,
                                    float(C) if adaptive else 0.0, _ptr(topk_ids), _ptr(topk_logq),
                                    _ptr(lse), _ptr(entropy), _ptr(lambda_d), _ptr(ws), nws,
                                    _ptr(dev_status), _stream(stream))
    _check(st, "presto_topk_entropy")
    return topk_ids, topk_logq, lse, entropy, lambda_d


def presto_topk_slots(slot_logits, accept_len, accept_path, slot_offset, L, k, node_token=None,
                      bonus=None, ctx2_next=None, topk_ids=None, topk_logq=None, lse=None, ws=None,
                      dev_status=None, stream=None, with_lse=True):
    """Top-k of the next round's drafter rows, read in place from the mask slots of
    the deepest accepted node (App. C (II)).  slot_logits [B, n_prev, n_slots, V]
    (unit last stride, packed); accept_len [B], accept_path [B, path_len] from
    presto_accept.  With node_token and bonus also returns ctx2_next [B, 2].
    Returns (topk_ids, topk_logq, lse, ctx2_next)."""
    if slot_logits.dim() != 4 or slot_logits.stride(3) != 1:
        raise ValueError("slot_logits must be [B, n_prev, n_slots, V] with unit last stride")
    B, n_prev, n_slots, V = slot_logits.shape
    rs = slot_logits.stride(2)
    if slot_logits.stride(1) != n_slots * rs or slot_logits.stride(0) != n_prev * n_slots * rs:
        raise ValueError("slot_logits rows must be packed")
    dtype = {torch.float32: PRESTO_F32, torch.bfloat16: PRESTO_BF16}.get(slot_logits.dtype)
    if dtype is None:
        raise ValueError("slot_logits must be float32 or bfloat16")
    dev = slot_logits.device
    path_len = accept_path.shape[1]
    _need(accept_len, torch.int32, (B,), "accept_len")
    _need(accept_path, torch.int32, (B, path_len), "accept_path")
    topk_ids = torch.empty(B, L, k, dtype=torch.int32, device=dev) if topk_ids is None else topk_ids
    topk_logq = torch.empty(B, L, k, dtype=torch.float32, device=dev) if topk_logq is None else topk_logq
    if lse is None and with_lse:
        lse = torch.empty(B, L, dtype=torch.float32, device=dev)
    if node_token is not None:
        _need(node_token, torch.int32, (B, n_prev), "node_token")
        _need(bonus, torch.int32, (B,), "bonus")
        if ctx2_next is None:
            ctx2_next = torch.empty(B, 2, dtype=torch.int32, device=dev)
        _need(ctx2_next, torch.int32, (B, 2), "ctx2_next")
    _need(topk_ids, torch.int32, (B, L, k), "topk_ids")
    _need(topk_logq, torch.float32, (B, L, k), "topk_logq")
    ws, nws = _ws(presto_topk_workspace(B, L, V, k), dev, ws)
    st = load().presto_topk_slots(_ptr(slot_logits), dtype, B, n_prev, n_slots, V, rs,
                                  _ptr(accept_len), _ptr(accept_path), path_len, slot_offset, L, k,
                                  _ptr(node_token), _ptr(bonus), _ptr(ctx2_next), _ptr(topk_ids),
                                  _ptr(topk_logq), _ptr(lse), _ptr(ws), nws, _ptr(dev_status),
                                  _stream(stream))
    _check(st, "presto_topk_slots")
    return topk_ids, topk_logq, lse, ctx2_next


# ------------------------------------------------------------------ trigram table

def pack_trigram_keys(a, b, t) -> np.ndarray:
    """Key layout of the table: (a << 36) | (b << 18) | t, as uint64."""
    a = np.asarray(a, np.uint64)
    b = np.asarray(b, np.uint64)
    t = np.asarray(t, np.uint64)
    return (a << np.uint64(36)) | (b << np.uint64(18)) | t


class Ngram3Table:
    """Device-resident trigram table (keys/logrho tensors + the C descriptor)."""

    def __init__(self, log2_cap: int, miss_logrho: float, device="cuda"):
        cap = 1 << log2_cap
        self.keys = torch.empty(cap, dtype=torch.int64, device=device)
        self.logrho = torch.zeros(cap, dtype=torch.float32, device=device)
        self.desc = Ngram3(self.keys.data_ptr(), self.logrho.data_ptr(), log2_cap, miss_logrho)
        self.log2_cap = log2_cap
        self.miss_logrho = miss_logrho

    def clear(self, stream=None):
        _check(load().presto_ngram3_clear(ctypes.byref(self.desc), _stream(stream)),
               "presto_ngram3_clear")

    def insert(self, keys, logrho, dev_status=None, stream=None):
        """keys: int64 tensor (uint64 bit patterns) on the device; logrho float32."""
        n = int(keys.numel())
        _check(load().presto_ngram3_insert(ctypes.byref(self.desc), _ptr(keys), _ptr(logrho), n,
                                           _ptr(dev_status), _stream(stream)),
               "presto_ngram3_insert")

    @classmethod
    def from_entries(cls, a, b, t, logrho, log2_cap, miss_logrho, device="cuda"):
        n = len(logrho)
        if n > (1 << log2_cap):
            raise ValueError(f"{n} entries do not fit 2^{log2_cap} slots")
        tab = cls(log2_cap, miss_logrho, device)
        tab.clear()
        keys = torch.from_numpy(pack_trigram_keys(a, b, t).view(np.int64)).to(device)
        vals = torch.from_numpy(np.asarray(logrho, np.float32)).to(device)
        st = torch.zeros(1, dtype=torch.int32, device=device)
        tab.insert(keys, vals, dev_status=st)
        if int(st.item()) != 0:
            raise PrestoError(f"trigram insert: {dev_status_names(int(st.item()))}")
        return tab


# ------------------------------------------------------------------ tree build

SEARCH_BEST_FIRST, SEARCH_BEAM, SEARCH_EAGER = 0, 1, 2


def presto_build_workspace(B, L, k, N, beam_width=1) -> int:
    return int(load().presto_build_workspace_ex(B, L, k, N, beam_width))


def presto_score_build_tree(topk_ids, topk_logq, ctx2, ngram, lam, N, b=None, out=None, ws=None,
                            dev_status=None, stream=None, lambda_d=None,
                            policy=SEARCH_BEST_FIRST, beam_width=1, kv_len=None, mask=None,
                            pos_ids=None):
    """Returns dict(token, parent, depth, score, n_nodes) of device tensors.
    ``lambda_d`` ([B, L] float32, optional) gives each drafter row its own lambda;
    ``policy`` is SEARCH_BEST_FIRST, SEARCH_BEAM (with ``beam_width``) or SEARCH_EAGER.
    With ``kv_len`` the same kernel also writes the tree mask and position ids
    (presto_score_build_tree_mask), returned as out["mask"], out["pos_ids"]."""
    B, L, k = topk_ids.shape
    b = k if b is None else b
    dev = topk_ids.device
    _need(topk_ids, torch.int32, (B, L, k), "topk_ids")
    _need(topk_logq, torch.float32, (B, L, k), "topk_logq")
    _need(ctx2, torch.int32, (B, 2), "ctx2")
    if lambda_d is not None:
        _need(lambda_d, torch.float32, (B, L), "lambda_d")
    if out is None:
        out = {"token": torch.empty(B, N, dtype=torch.int32, device=dev),
               "parent": torch.empty(B, N, dtype=torch.int32, device=dev),
               "depth": torch.empty(B, N, dtype=torch.int32, device=dev),
               "score": torch.empty(B, N, dtype=torch.float32, device=dev),
               "n_nodes": torch.empty(B, dtype=torch.int32, device=dev)}
    ws, nws = _ws(presto_build_workspace(B, L, k, N, beam_width), dev, ws)
    desc = None if ngram is None else ctypes.byref(ngram.desc)
    if kv_len is not None:
        W = (N + 31) // 32
        _need(kv_len, torch.int32, (B,), "kv_len")
        mask = torch.empty(B, N, W, dtype=torch.int32, device=dev) if mask is None else mask
        pos_ids = torch.empty(B, N, dtype=torch.int32, device=dev) if pos_ids is None else pos_ids
        _need(mask, torch.int32, (B, N, W), "mask")
        _need(pos_ids, torch.int32, (B, N), "pos_ids")
        out["mask"], out["pos_ids"] = mask, pos_ids
    st = load().presto_score_build_tree_mask(
        _ptr(topk_ids), _ptr(topk_logq), B, L, k, b, _ptr(ctx2), desc, float(lam),
        _ptr(lambda_d), int(policy), int(beam_width), N,
        _ptr(out["token"]), _ptr(out["parent"]), _ptr(out["depth"]), _ptr(out["score"]),
        _ptr(out["n_nodes"]), _ptr(kv_len), _ptr(mask) if kv_len is not None else None,
        _ptr(pos_ids) if kv_len is not None else None, _ptr(ws), nws, _ptr(dev_status),
        _stream(stream))
    _check(st, "presto_score_build_tree_mask")
    return out


def presto_score_build_tree_noalloc(topk_ids, topk_logq, ctx2, ngram, lam, N, out, b=None,
                                    dev_status=None, stream=None, lambda_d=None,
                                    policy=SEARCH_BEST_FIRST, beam_width=1, kv_len=None,
                                    mask=None, pos_ids=None):
    """presto_score_build_tree without a workspace, for callers that cannot allocate
    device memory: the library keeps the build's scratch in a fixed 1 MiB device
    array shared by every call on the device (calls that may overlap on the GPU
    race).  Outputs are passed in (``out`` as presto_score_build_tree returns it,
    plus mask and pos_ids with kv_len): nothing is allocated here either."""
    B, L, k = topk_ids.shape
    b = k if b is None else b
    _need(topk_ids, torch.int32, (B, L, k), "topk_ids")
    _need(topk_logq, torch.float32, (B, L, k), "topk_logq")
    _need(ctx2, torch.int32, (B, 2), "ctx2")
    for key, dt, shape in (("token", torch.int32, (B, N)), ("parent", torch.int32, (B, N)),
                           ("depth", torch.int32, (B, N)), ("score", torch.float32, (B, N)),
                           ("n_nodes", torch.int32, (B,))):
        _need(out[key], dt, shape, key)
    if kv_len is not None:
        W = (N + 31) // 32
        _need(kv_len, torch.int32, (B,), "kv_len")
        _need(mask, torch.int32, (B, N, W), "mask")
        _need(pos_ids, torch.int32, (B, N), "pos_ids")
    desc = None if ngram is None else ctypes.byref(ngram.desc)
    st = load().presto_score_build_tree_noalloc(
        _ptr(topk_ids), _ptr(topk_logq), B, L, k, b, _ptr(ctx2), desc, float(lam),
        _ptr(lambda_d), int(policy), int(beam_width), N,
        _ptr(out["token"]), _ptr(out["parent"]), _ptr(out["depth"]), _ptr(out["score"]),
        _ptr(out["n_nodes"]), _ptr(kv_len), _ptr(mask), _ptr(pos_ids), _ptr(dev_status),
        _stream(stream))
    _check(st, "presto_score_build_tree_noalloc")
    return out


# ------------------------------------------------------------------ mask / attention / accept

def presto_tree_mask(node_parent, node_depth, n_nodes, kv_len, mask=None, pos_ids=None,
                     dev_status=None, stream=None):
    B, N = node_parent.shape
    W = (N + 31) // 32
    dev = node_parent.device
    mask = torch.empty(B, N, W, dtype=torch.int32, device=dev) if mask is None else mask
    pos_ids = torch.empty(B, N, dtype=torch.int32, device=dev) if pos_ids is None else pos_ids
    for t, name in ((node_parent, "node_parent"), (node_depth, "node_depth")):
        _need(t, torch.int32, (B, N), name)
    _need(n_nodes, torch.int32, (B,), "n_nodes")
    _need(kv_len, torch.int32, (B,), "kv_len")
    st = load().presto_tree_mask(_ptr(node_parent), _ptr(node_depth), _ptr(n_nodes), _ptr(kv_len),
                                 B, N, _ptr(mask), _ptr(pos_ids), _ptr(dev_status), _stream(stream))
    _check(st, "presto_tree_mask")
    return mask, pos_ids


def presto_attn_workspace(B, N, Hq, Hkv, D, Tmax) -> int:
    return int(load().presto_attn_workspace(B, N, Hq, Hkv, D, Tmax))


def presto_attn_launches(B, N, Hq, Hkv, D, Tmax) -> int:
    """Kernels one presto_tree_attention call of these shapes launches (0: refused)."""
    return int(load().presto_attn_launches(B, N, Hq, Hkv, D, Tmax))


def presto_tree_attention(q, k_cache, v_cache, kv_len, k_tree, v_tree, mask, n_nodes,
                          sm_scale=None, out=None, lse=None, ws=None, dev_status=None,
                          stream=None, with_lse=True):
    B, N, Hq, D = q.shape
    Hkv, Tmax = k_cache.shape[1], k_cache.shape[2]
    dev = q.device
    bf = torch.bfloat16
    _need(q, bf, (B, N, Hq, D), "q")
    _need(k_cache, bf, (B, Hkv, Tmax, D), "k_cache")
    _need(v_cache, bf, (B, Hkv, Tmax, D), "v_cache")
    _need(k_tree, bf, (B, N, Hkv, D), "k_tree")
    _need(v_tree, bf, (B, N, Hkv, D), "v_tree")
    _need(kv_len, torch.int32, (B,), "kv_len")
    _need(n_nodes, torch.int32, (B,), "n_nodes")
    sm_scale = 1.0 / float(D) ** 0.5 if sm_scale is None else sm_scale
    out = torch.empty(B, N, Hq, D, dtype=bf, device=dev) if out is None else out
    if lse is None and with_lse:
        lse = torch.empty(B, N, Hq, dtype=torch.float32, device=dev)
    ws, nws = _ws(presto_attn_workspace(B, N, Hq, Hkv, D, Tmax), dev, ws)
    st = load().presto_tree_attention(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(kv_len), Tmax, _ptr(k_tree), _ptr(v_tree),
        _ptr(mask), _ptr(n_nodes), B, N, Hq, Hkv, D, float(sm_scale), _ptr(out), _ptr(lse),
        _ptr(ws), nws, _ptr(dev_status), _stream(stream))
    _check(st, "presto_tree_attention")
    return out, lse


def presto_accept(node_token, node_parent, node_depth, mask, n_nodes, target_token, L,
                  accept_len=None, accept_path=None, bonus=None, dev_status=None, stream=None):
    B, N = node_token.shape
    dev = node_token.device
    accept_len = torch.empty(B, dtype=torch.int32, device=dev) if accept_len is None else accept_len
    accept_path = (torch.empty(B, L + 1, dtype=torch.int32, device=dev)
                   if accept_path is None else accept_path)
    bonus = torch.empty(B, dtype=torch.int32, device=dev) if bonus is None else bonus
    _need(target_token, torch.int32, (B, N), "target_token")
    st = load().presto_accept(_ptr(node_token), _ptr(node_parent), _ptr(node_depth), _ptr(mask),
                              _ptr(n_nodes), _ptr(target_token), B, N, L, _ptr(accept_len),
                              _ptr(accept_path), _ptr(bonus), _ptr(dev_status), _stream(stream))
    _check(st, "presto_accept")
    return accept_len, accept_path, bonus


def presto_build_flags() -> int:
    """Flags of the loaded library (BUILD_CHECKS for the bounds-checked debug build)."""
    return int(load().presto_build_flags())


def presto_selftest_wait_timeout(dev_status, wait_cycles, stream=None):
    """One GPU thread waits wait_cycles SM cycles for a barrier phase nothing
    completes; PRESTO_DEV_TIMEOUT is ORed into dev_status (a device int32 tensor)."""
    _need(dev_status, torch.int32, (1,), "dev_status")
    _check(load().presto_selftest_wait_timeout(_ptr(dev_status), int(wait_cycles), _stream(stream)),
           "presto_selftest_wait_timeout")

"""Python binding of the SEED draft/verify attention library (include/seed.h).

Argument marshalling only: every call checks that its torch tensors have the
dtype, device, shape and layout the C ABI expects, passes their data pointers
and the current CUDA stream to ``libseed.so``, and raises on a non-OK status.
All arithmetic runs in the library's CUDA kernels; there is no fallback, and
every entry point fails loudly when the library has not been built.

Entry points carry the C names: seed_workspace_bytes, seed_draft_kv_append,
seed_draft_attn, seed_kv_append, seed_verify_attn, seed_accept_commit, and
seed_verify_attn_noalloc (verify attention on the library's built-in scratch,
for callers that cannot provide a workspace), and the tree-verification calls
seed_tree_verify_attn, seed_tree_accept_commit, seed_tree_kv_compact, the
dynamic-drafting head seed_draft_head_topk, and the draft step on the device:
seed_linear, seed_embed, seed_rmsnorm and seed_draft_layer, and the decoder's
block-causal training attention seed_block_attn.
"""

from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libseed.so")

SEED_OK = 0
SEED_ERR_SCRATCH_LIMIT = 7
NOALLOC_SCRATCH_BYTES = 32 << 20   # SEED_NOALLOC_SCRATCH_BYTES of seed.h
DEVERR = {1: "ctx_len", 2: "draft_len", 4: "n_q", 8: "page", 16: "k_b", 32: "workspace",
          64: "timeout", 128: "tree", 256: "token"}
MAX_KMAX = 31


class _Cfg(ctypes.Structure):
    _fields_ = [("hq", ctypes.c_int32), ("hkv", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("kmax", ctypes.c_int32), ("scale", ctypes.c_float)]


class _Layer(ctypes.Structure):
    _fields_ = [("d_model", ctypes.c_int32), ("d_ff", ctypes.c_int32),
                ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float)] + [
        (n, ctypes.c_void_p) for n in ("g_attn", "w_qkv", "g_q", "g_k", "w_o", "g_mlp", "w_gate",
                                       "w_up", "w_down")]


class _KV(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("page_table", ctypes.c_void_p),
                ("max_pages", ctypes.c_int32), ("num_pages", ctypes.c_int32)]


_P = ctypes.c_void_p
_I = ctypes.c_int32
_SIGS = {
    "seed_abi_version": (_I, []),
    "seed_status_string": (ctypes.c_char_p, [_I]),
    "seed_workspace_bytes": (ctypes.c_size_t, [ctypes.POINTER(_Cfg), _I]),
    "seed_attn_route": (_I, [ctypes.POINTER(_Cfg), _I, _I, _I]),
    "seed_draft_kv_append": (_I, [ctypes.POINTER(_Cfg), _I, _P, _P, _P, _P, _P, _P, _P]),
    "seed_draft_attn": (_I, [ctypes.POINTER(_Cfg), _I, _P, _KV, _P, _P, _P, _P, _P, _P, _P,
                             ctypes.c_size_t, _P, _P]),
    "seed_kv_append": (_I, [ctypes.POINTER(_Cfg), _I, _KV, _P, _P, _P, _P, _P, _P]),
    "seed_verify_attn": (_I, [ctypes.POINTER(_Cfg), _I, _P, _P, _KV, _P, _P, _P, _P,
                              ctypes.c_size_t, _P, _P]),
    "seed_accept_commit": (_I, [_I, _I, _P, _P, _P, _P, _I, _I, _P, _P, _P, _P, _P, _P]),
    "seed_verify_attn_noalloc": (_I, [ctypes.POINTER(_Cfg), _I, _P, _P, _KV, _P, _P, _P, _P,
                                      _P]),
    "seed_tree_verify_attn": (_I, [ctypes.POINTER(_Cfg), _I, _P, _P, _P, _KV, _P, _P, _P, _P,
                                   ctypes.c_size_t, _P, _P]),
    "seed_tree_accept_commit": (_I, [_I, _I, _P, _P, _P, _P, _P, _I, _I, _P, _P, _P, _P, _P,
                                     _P, _P]),
    "seed_tree_kv_compact": (_I, [ctypes.POINTER(_Cfg), _I, _KV, _P, _P, _P, _P, _P]),
    "seed_draft_head_workspace_bytes": (ctypes.c_size_t, [_I]),
    "seed_linear_workspace_bytes": (ctypes.c_size_t, [_I, _I, _I, _I]),
    "seed_linear": (_I, [_I, _I, _I, _P, _P, _P, _I, _P, _P, ctypes.c_size_t, _P, _P]),
    "seed_embed": (_I, [_I, _I, _I, _P, _P, _P, _P, _P]),
    "seed_rmsnorm": (_I, [_I, _I, _P, _P, ctypes.c_float, _P, _P]),
    "seed_draft_layer_workspace_bytes": (ctypes.c_size_t, [ctypes.POINTER(_Cfg),
                                                           ctypes.POINTER(_Layer), _I]),
    "seed_draft_layer": (_I, [ctypes.POINTER(_Cfg), _I, ctypes.POINTER(_Layer), _P, _KV, _P, _P,
                              _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "seed_block_attn_workspace_bytes": (ctypes.c_size_t, [ctypes.POINTER(_Cfg), _I, _I, _I]),
    "seed_block_attn": (_I, [ctypes.POINTER(_Cfg), _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P,
                             ctypes.c_size_t, _P, _P]),
    "seed_draft_head_topk": (_I, [_I, _I, _I, _P, _P, ctypes.c_float, _P, _P, _P, _P, _P, _P,
                                  ctypes.c_size_t, _P, _P]),
}


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            f"{LIB_PATH} is missing: build it with `python -m paper_2609_36590_gb300.build` "
            "(the SEED path has no CPU fallback)")
    lib = ctypes.CDLL(LIB_PATH)
    for name, (res, args) in _SIGS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


class _Lazy:
    """Loads libseed.so on first use, so that the build script can import the
    package before the library exists; every entry point fails loudly if it is
    still missing then."""

    _cdll = None

    def __getattr__(self, name):
        if _Lazy._cdll is None:
            _Lazy._cdll = _load()
        return getattr(_Lazy._cdll, name)


_lib = _Lazy()


class SeedError(RuntimeError):
    pass


def _check(status: int) -> None:
    if status != SEED_OK:
        msg = _lib.seed_status_string(status).decode()
        raise SeedError(f"libseed status {status}: {msg}")


@dataclass(frozen=True)
class SeedConfig:
    hq: int
    hkv: int
    head_dim: int
    kmax: int
    page_size: int = 16
    scale: float = 0.0

    def c(self) -> _Cfg:
        return _Cfg(self.hq, self.hkv, self.head_dim, self.page_size, self.kmax, self.scale)


@dataclass
class PagedKV:
    """One layer's cache: k, v bf16 [num_pages, hkv, page_size, head_dim];
    page_table int32 [batch, max_pages]."""
    k: torch.Tensor
    v: torch.Tensor
    page_table: torch.Tensor

    def c(self) -> _KV:
        return _KV(self.k.data_ptr(), self.v.data_ptr(), self.page_table.data_ptr(),
                   self.page_table.shape[1], self.k.shape[0])


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _t(x: torch.Tensor, dtype, shape, name: str) -> int:
    if not isinstance(x, torch.Tensor):
        raise TypeError(f"{name}: expected a torch.Tensor")
    if x.dtype != dtype:
        raise TypeError(f"{name}: dtype {x.dtype}, expected {dtype}")
    if not x.is_cuda:
        raise ValueError(f"{name}: must be a CUDA tensor")
    if not x.is_contiguous():
        raise ValueError(f"{name}: must be contiguous")
    if shape is not None and tuple(x.shape) != tuple(shape):
        raise ValueError(f"{name}: shape {tuple(x.shape)}, expected {tuple(shape)}")
    return x.data_ptr()


def _kv_checked(cfg: SeedConfig, kv: PagedKV, batch: int) -> _KV:
    shp = (kv.k.shape[0], cfg.hkv, cfg.page_size, cfg.head_dim)
    _t(kv.k, torch.bfloat16, shp, "kv.k")
    _t(kv.v, torch.bfloat16, shp, "kv.v")
    _t(kv.page_table, torch.int32, (batch, kv.page_table.shape[1]), "kv.page_table")
    return kv.c()


def seed_workspace_bytes(cfg: SeedConfig, batch: int) -> int:
    c = cfg.c()
    n = _lib.seed_workspace_bytes(ctypes.byref(c), batch)
    if n == 0:
        raise SeedError("invalid configuration")
    return int(n)


ROUTE_CUDA_CORE, ROUTE_TC_ROWS, ROUTE_TC_KEYS = 0, 1, 2
ROUTE_KERNELS = {0: "decode_attn_kernel", 1: "attn_tc_kernel", 2: "attn_kt_kernel",
                 8: "attn_cl_kernel", 12: "attn_cl_kernel", 16: "attn_cl_kernel"}


def seed_attn_route(cfg: SeedConfig, batch: int, draft: bool, max_pages: int) -> int:
    """The kernel seed_draft_attn (draft) or seed_verify_attn runs for this
    shape on the current device: ROUTE_* or a cluster size 8, 12, 16."""
    r = _lib.seed_attn_route(ctypes.byref(cfg.c()), batch, 1 if draft else 0, max_pages)
    if r < 0:
        raise SeedError(f"seed_attn_route: invalid arguments ({r})")
    return r


def new_workspace(cfg: SeedConfig, batch: int, device=None) -> torch.Tensor:
    """A zero-filled workspace (uint8) for seed_draft_attn / seed_verify_attn."""
    return torch.zeros(seed_workspace_bytes(cfg, batch), dtype=torch.uint8, device=device or "cuda")


def seed_draft_kv_append(cfg: SeedConfig, k_new, v_new, draft_lens, draft_k, draft_v, err,
                         stream=None) -> None:
    B = draft_lens.shape[0]
    c = cfg.c()
    _check(_lib.seed_draft_kv_append(
        ctypes.byref(c), B,
        _t(k_new, torch.bfloat16, (B, cfg.hkv, cfg.head_dim), "k_new"),
        _t(v_new, torch.bfloat16, (B, cfg.hkv, cfg.head_dim), "v_new"),
        _t(draft_lens, torch.int32, (B,), "draft_lens"),
        _t(draft_k, torch.bfloat16, (B, cfg.hkv, cfg.kmax, cfg.head_dim), "draft_k"),
        _t(draft_v, torch.bfloat16, (B, cfg.hkv, cfg.kmax, cfg.head_dim), "draft_v"),
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


def seed_draft_attn(cfg: SeedConfig, q, ctx_kv: PagedKV, draft_k, draft_v, ctx_lens, draft_lens,
                    out, lse, ws, err, stream=None) -> None:
    B = q.shape[0]
    c = cfg.c()
    _check(_lib.seed_draft_attn(
        ctypes.byref(c), B,
        _t(q, torch.bfloat16, (B, cfg.hq, cfg.head_dim), "q"),
        _kv_checked(cfg, ctx_kv, B),
        _t(draft_k, torch.bfloat16, (B, cfg.hkv, cfg.kmax, cfg.head_dim), "draft_k"),
        _t(draft_v, torch.bfloat16, (B, cfg.hkv, cfg.kmax, cfg.head_dim), "draft_v"),
        _t(ctx_lens, torch.int32, (B,), "ctx_lens"),
        _t(draft_lens, torch.int32, (B,), "draft_lens"),
        _t(out, torch.float32, (B, cfg.hq, cfg.head_dim), "out"),
        _t(lse, torch.float32, (B, cfg.hq), "lse") if lse is not None else None,
        _t(ws, torch.uint8, None, "ws"), ws.numel(),
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


def seed_kv_append(cfg: SeedConfig, kv: PagedKV, k_new, v_new, n_new, ctx_lens, err,
                   stream=None) -> None:
    B = n_new.shape[0]
    c = cfg.c()
    shp = (B, cfg.kmax + 1, cfg.hkv, cfg.head_dim)
    _check(_lib.seed_kv_append(
        ctypes.byref(c), B, _kv_checked(cfg, kv, B),
        _t(k_new, torch.bfloat16, shp, "k_new"), _t(v_new, torch.bfloat16, shp, "v_new"),
        _t(n_new, torch.int32, (B,), "n_new"), _t(ctx_lens, torch.int32, (B,), "ctx_lens"),
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


def seed_verify_attn(cfg: SeedConfig, q, n_q, kv: PagedKV, ctx_lens, out, lse, ws, err,
                     stream=None) -> None:
    B = q.shape[0]
    c = cfg.c()
    W = cfg.kmax + 1
    _check(_lib.seed_verify_attn(
        ctypes.byref(c), B,
        _t(q, torch.bfloat16, (B, W, cfg.hq, cfg.head_dim), "q"),
        _t(n_q, torch.int32, (B,), "n_q"),
        _kv_checked(cfg, kv, B),
        _t(ctx_lens, torch.int32, (B,), "ctx_lens"),
        _t(out, torch.float32, (B, W, cfg.hq, cfg.head_dim), "out"),
        _t(lse, torch.float32, (B, W, cfg.hq), "lse") if lse is not None else None,
        _t(ws, torch.uint8, None, "ws"), ws.numel(),
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


def seed_verify_attn_noalloc(cfg: SeedConfig, q, n_q, kv: PagedKV, ctx_lens, out, lse, err,
                             stream=None) -> None:
    """seed_verify_attn without a workspace argument: the library uses its
    built-in per-device scratch. Calls that overlap in time on one device race
    on that scratch; issue them on one stream."""
    B = q.shape[0]
    c = cfg.c()
    W = cfg.kmax + 1
    _check(_lib.seed_verify_attn_noalloc(
        ctypes.byref(c), B,
        _t(q, torch.bfloat16, (B, W, cfg.hq, cfg.head_dim), "q"),
        _t(n_q, torch.int32, (B,), "n_q"),
        _kv_checked(cfg, kv, B),
        _t(ctx_lens, torch.int32, (B,), "ctx_lens"),
        _t(out, torch.float32, (B, W, cfg.hq, cfg.head_dim), "out"),
        _t(lse, torch.float32, (B, W, cfg.hq), "lse") if lse is not None else None,
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


def seed_tree_verify_attn(cfg: SeedConfig, q, n_nodes, anc, kv: PagedKV, ctx_lens, out, lse, ws,
                          err, stream=None) -> None:
    """Verify attention over draft trees (tree-structured mask); anc is int32
    holding the uint32 ancestor bit masks [B, kmax+1]."""
    B = q.shape[0]
    c = cfg.c()
    W = cfg.kmax + 1
    _check(_lib.seed_tree_verify_attn(
        ctypes.byref(c), B,
        _t(q, torch.bfloat16, (B, W, cfg.hq, cfg.head_dim), "q"),
        _t(n_nodes, torch.int32, (B,), "n_nodes"),
        _t(anc, torch.int32, (B, W), "anc"),
        _kv_checked(cfg, kv, B),
        _t(ctx_lens, torch.int32, (B,), "ctx_lens"),
        _t(out, torch.float32, (B, W, cfg.hq, cfg.head_dim), "out"),
        _t(lse, torch.float32, (B, W, cfg.hq), "lse") if lse is not None else None,
        _t(ws, torch.uint8, None, "ws"), ws.numel(),
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


def seed_tree_accept_commit(kmax: int, tok, parent, n_nodes, target_ids, page_table,
                            page_size: int, ctx_lens, accepted, tokens, path, committed_slots,
                            err, stream=None) -> None:
    B = n_nodes.shape[0]
    W = kmax + 1
    _check(_lib.seed_tree_accept_commit(
        B, kmax,
        _t(tok, torch.int32, (B, W), "tok"),
        _t(parent, torch.int32, (B, W), "parent"),
        _t(n_nodes, torch.int32, (B,), "n_nodes"),
        _t(target_ids, torch.int32, (B, W), "target_ids"),
        _t(page_table, torch.int32, (B, page_table.shape[1]), "page_table"),
        page_table.shape[1], page_size,
        _t(ctx_lens, torch.int32, (B,), "ctx_lens"),
        _t(accepted, torch.int32, (B,), "accepted"),
        _t(tokens, torch.int32, (B, W), "tokens"),
        _t(path, torch.int32, (B, W), "path"),
        _t(committed_slots, torch.int32, (B, W), "committed_slots"),
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


def seed_tree_kv_compact(cfg: SeedConfig, kv: PagedKV, path, accepted, ctx_lens, err,
                         stream=None) -> None:
    B = accepted.shape[0]
    c = cfg.c()
    _check(_lib.seed_tree_kv_compact(
        ctypes.byref(c), B, _kv_checked(cfg, kv, B),
        _t(path, torch.int32, (B, cfg.kmax + 1), "path"),
        _t(accepted, torch.int32, (B,), "accepted"),
        _t(ctx_lens, torch.int32, (B,), "ctx_lens"),
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


def new_draft_head_workspace(batch: int, device=None) -> torch.Tensor:
    n = _lib.seed_draft_head_workspace_bytes(batch)
    if n == 0:
        raise SeedError("batch outside the supported range")
    return torch.empty(int(n), dtype=torch.uint8, device=device or "cuda")


def seed_draft_head_topk(h, w_out, tau: float, ids, probs, n_sib, stop, lse, ws, err,
                         stream=None) -> None:
    """LM head + softmax + top-10 per sequence, sibling count and stop flag."""
    B, d = h.shape
    V = w_out.shape[0]
    _check(_lib.seed_draft_head_topk(
        B, d, V,
        _t(h, torch.bfloat16, (B, d), "h"),
        _t(w_out, torch.bfloat16, (V, d), "w_out"),
        float(tau),
        _t(ids, torch.int32, (B, 10), "ids"),
        _t(probs, torch.float32, (B, 10), "probs"),
        _t(n_sib, torch.int32, (B,), "n_sib"),
        _t(stop, torch.int32, (B,), "stop"),
        _t(lse, torch.float32, (B,), "lse") if lse is not None else None,
        _t(ws, torch.uint8, None, "ws"), ws.numel(),
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


def seed_accept_commit(kmax: int, draft_ids, target_ids, k_b, page_table, page_size: int,
                       ctx_lens, accepted, tokens, committed_slots, err, stream=None) -> None:
    B = k_b.shape[0]
    _check(_lib.seed_accept_commit(
        B, kmax,
        _t(draft_ids, torch.int32, (B, kmax), "draft_ids"),
        _t(target_ids, torch.int32, (B, kmax + 1), "target_ids"),
        _t(k_b, torch.int32, (B,), "k_b"),
        _t(page_table, torch.int32, (B, page_table.shape[1]), "page_table"),
        page_table.shape[1], page_size,
        _t(ctx_lens, torch.int32, (B,), "ctx_lens"),
        _t(accepted, torch.int32, (B,), "accepted"),
        _t(tokens, torch.int32, (B, kmax + 1), "tokens"),
        _t(committed_slots, torch.int32, (B, kmax + 1), "committed_slots"),
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


LINEAR_F32, LINEAR_RESID_F32, LINEAR_SWIGLU = 0, 1, 2


def new_linear_workspace(batch: int, n_out: int, k_in: int, epilogue: int,
                         device=None) -> torch.Tensor:
    """A zero-filled workspace for seed_linear with these sizes."""
    n = _lib.seed_linear_workspace_bytes(batch, n_out, k_in, epilogue)
    if n == 0:
        raise SeedError("invalid seed_linear sizes")
    return torch.zeros(int(n), dtype=torch.uint8, device=device or "cuda")


def seed_linear(x, w, y, ws, err, epilogue: int = LINEAR_F32, w2=None, stream=None) -> None:
    """y (epilogue) x w^T: x bf16 [B, K], w (and w2 for SwiGLU) bf16 [N, K];
    y f32 [B, N] (F32, RESID_F32) or bf16 [B, N] (SWIGLU)."""
    B, K = x.shape
    N = w.shape[0]
    ydt = torch.bfloat16 if epilogue == LINEAR_SWIGLU else torch.float32
    _check(_lib.seed_linear(
        B, K, N, _t(x, torch.bfloat16, (B, K), "x"), _t(w, torch.bfloat16, (N, K), "w"),
        _t(w2, torch.bfloat16, (N, K), "w2") if w2 is not None else None, epilogue,
        _t(y, ydt, (B, N), "y"), _t(ws, torch.uint8, None, "ws"), ws.numel(),
        _t(err, torch.int32, (1,), "err"), _stream(stream)))


def seed_embed(tokens, w_emb, x, err, stream=None) -> None:
    B = tokens.shape[0]
    V, d = w_emb.shape
    _check(_lib.seed_embed(B, d, V, _t(tokens, torch.int32, (B,), "tokens"),
                           _t(w_emb, torch.bfloat16, (V, d), "w_emb"),
                           _t(x, torch.float32, (B, d), "x"), _t(err, torch.int32, (1,), "err"),
                           _stream(stream)))


def seed_rmsnorm(x, gamma, eps: float, y, stream=None) -> None:
    rows, n = x.shape
    _check(_lib.seed_rmsnorm(rows, n, _t(x, torch.float32, (rows, n), "x"),
                             _t(gamma, torch.bfloat16, (n,), "gamma"), eps,
                             _t(y, torch.bfloat16, (rows, n), "y"), _stream(stream)))


@dataclass
class DecoderLayer:
    """One decoder layer's bf16 weights (nn.Linear layout) for seed_draft_layer."""
    g_attn: torch.Tensor
    w_qkv: torch.Tensor
    g_q: torch.Tensor
    g_k: torch.Tensor
    w_o: torch.Tensor
    g_mlp: torch.Tensor
    w_gate: torch.Tensor
    w_up: torch.Tensor
    w_down: torch.Tensor
    rms_eps: float = 1e-6
    rope_theta: float = 1e6

    def c(self, cfg: SeedConfig) -> _Layer:
        dm, F = self.w_gate.shape[1], self.w_gate.shape[0]
        D, nqkv = cfg.head_dim, (cfg.hq + 2 * cfg.hkv) * cfg.head_dim
        shapes = dict(g_attn=(dm,), w_qkv=(nqkv, dm), g_q=(D,), g_k=(D,), w_o=(dm, cfg.hq * D),
                      g_mlp=(dm,), w_gate=(F, dm), w_up=(F, dm), w_down=(dm, F))
        ptr = {n: _t(getattr(self, n), torch.bfloat16, shp, n) for n, shp in shapes.items()}
        return _Layer(dm, F, self.rms_eps, self.rope_theta, *[ptr[n] for n in shapes])


def new_draft_layer_workspace(cfg: SeedConfig, layer: DecoderLayer, batch: int,
                              device=None) -> torch.Tensor:
    c, lc = cfg.c(), layer.c(cfg)
    n = _lib.seed_draft_layer_workspace_bytes(ctypes.byref(c), ctypes.byref(lc), batch)
    if n == 0:
        raise SeedError("invalid seed_draft_layer configuration")
    return torch.zeros(int(n), dtype=torch.uint8, device=device or "cuda")


def seed_draft_layer(cfg: SeedConfig, layer: DecoderLayer, x, ctx_kv: PagedKV, ctx_lens, draft_k,
                     draft_v, draft_lens, ws, err, stream=None) -> None:
    B, dm = x.shape
    c, lc = cfg.c(), layer.c(cfg)
    _check(_lib.seed_draft_layer(
        ctypes.byref(c), B, ctypes.byref(lc), _t(x, torch.float32, (B, dm), "x"),
        _kv_checked(cfg, ctx_kv, B), _t(ctx_lens, torch.int32, (B,), "ctx_lens"),
        _t(draft_k, torch.bfloat16, (B, cfg.hkv, cfg.kmax, cfg.head_dim), "draft_k"),
        _t(draft_v, torch.bfloat16, (B, cfg.hkv, cfg.kmax, cfg.head_dim), "draft_v"),
        _t(draft_lens, torch.int32, (B,), "draft_lens"), _t(ws, torch.uint8, None, "ws"),
        ws.numel(), _t(err, torch.int32, (1,), "err"), _stream(stream)))


def new_block_attn_workspace(cfg: SeedConfig, batch: int, n: int, block: int,
                             device=None) -> torch.Tensor:
    c = cfg.c()
    nb = _lib.seed_block_attn_workspace_bytes(ctypes.byref(c), batch, n, block)
    if nb == 0:
        raise SeedError("invalid seed_block_attn sizes")
    return torch.zeros(int(nb), dtype=torch.uint8, device=device or "cuda")


def seed_block_attn(cfg: SeedConfig, block: int, q, k_dec, v_dec, k_spec, v_spec, out, lse, ws,
                    err, stream=None) -> None:
    """Block-causal training attention: q bf16 [B, n, hq, D]; k/v_dec and
    k/v_spec bf16 [B, n, hkv, D]; out f32 [B, n, hq, D]; lse f32 [B, n, hq]
    or None; ws uint8 (None on the tensor-core route, which uses none)."""
    B, n = q.shape[0], q.shape[1]
    kshape = (B, n, cfg.hkv, cfg.head_dim)
    c = cfg.c()
    _check(_lib.seed_block_attn(
        ctypes.byref(c), B, n, block, _t(q, torch.bfloat16, (B, n, cfg.hq, cfg.head_dim), "q"),
        _t(k_dec, torch.bfloat16, kshape, "k_dec"), _t(v_dec, torch.bfloat16, kshape, "v_dec"),
        _t(k_spec, torch.bfloat16, kshape, "k_spec"), _t(v_spec, torch.bfloat16, kshape, "v_spec"),
        _t(out, torch.float32, (B, n, cfg.hq, cfg.head_dim), "out"),
        _t(lse, torch.float32, (B, n, cfg.hq), "lse") if lse is not None else None,
        _t(ws, torch.uint8, None, "ws") if ws is not None else None,
        ws.numel() if ws is not None else 0, _t(err, torch.int32, (1,), "err"),
        _stream(stream)))


def library() -> ctypes.CDLL:
    """The loaded libseed.so (for ABI-level tests)."""
    if _Lazy._cdll is None:
        _Lazy._cdll = _load()
    return _Lazy._cdll

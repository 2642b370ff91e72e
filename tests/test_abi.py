"""The C ABI without a GPU: libseed.so loads, exports every function that
include/seed.h declares, and its host-side checks return the documented
statuses before touching CUDA (null pointers, unsupported shapes, bad page
ranges, small or misaligned workspaces, empty batches)."""

import ctypes
import os
import re
import subprocess

import pytest

import paper_2609_36590_gb300 as seed
from paper_2609_36590_gb300 import _Cfg, _KV, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "seed.h")

OK, ERR_NULL, ERR_SHAPE, ERR_RANGE, ERR_UNSUP, ERR_CUDA, ERR_WS = range(7)


@pytest.fixture(scope="module")
def lib():
    build.build()
    return seed.library()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(seed_[a-z_]+)\s*\(", text)))


def test_exports_every_declared_function(lib):
    names = declared_functions()
    assert len(names) >= 8
    out = subprocess.run(["nm", "-D", "--defined-only", seed.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (seed_\w+)", out))
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    for n in names:
        assert hasattr(lib, n)


def test_version_and_strings(lib):
    assert lib.seed_abi_version() == 4
    for s in range(7):
        assert len(lib.seed_status_string(s)) > 0
    assert lib.seed_status_string(99) == b"unknown status"


def cfg(**kw):
    base = dict(hq=32, hkv=8, head_dim=128, page_size=16, kmax=4, scale=0.0)
    base.update(kw)
    return _Cfg(**base)


@pytest.mark.parametrize("kw,expect", [
    (dict(), OK), (dict(head_dim=96), ERR_UNSUP), (dict(hq=24, hkv=8), ERR_UNSUP),
    (dict(hq=30, hkv=8), ERR_SHAPE), (dict(kmax=0), ERR_SHAPE), (dict(kmax=32), ERR_SHAPE), (dict(kmax=31), OK),
    (dict(page_size=32), ERR_UNSUP), (dict(scale=-1.0), ERR_SHAPE), (dict(head_dim=64), OK),
])
def test_workspace_bytes_validates_cfg(lib, kw, expect):
    c = cfg(**kw)
    n = lib.seed_workspace_bytes(ctypes.byref(c), 4)
    assert (n > 0) == (expect == OK)


def test_attn_route_host_logic(lib):
    """seed_attn_route rejects bad arguments and picks the CUDA-core and
    keys-as-rows routes by shape alone (the cluster route needs a GPU)."""
    def r(c, batch, draft, max_pages):
        return lib.seed_attn_route(ctypes.byref(c), batch, draft, max_pages)
    assert r(cfg(head_dim=96), 1, 0, 10) == -1
    assert r(cfg(), 0, 0, 10) == -1
    assert r(cfg(), 1, 0, 0) == -1
    assert r(cfg(head_dim=64, hq=8, hkv=2), 4, 0, 100) == 2            # 4 x 5 rows <= 48
    assert r(cfg(head_dim=64, hq=8, hkv=2), 4, 1, 100) == 2            # draft: 4 rows
    assert r(cfg(head_dim=64, hq=64, hkv=8, kmax=8), 4, 0, 100) == 0   # 8 x 9 = 72 rows
    assert r(cfg(), 64, 0, 4000) == 1                                   # 512 pairs


def test_workspace_grows_with_batch(lib):
    c = cfg()
    sizes = [lib.seed_workspace_bytes(ctypes.byref(c), b) for b in (1, 16, 64)]
    assert sizes[0] < sizes[1] < sizes[2]
    assert all(s % 256 == 0 for s in sizes)


FAKE = 0x10000  # never dereferenced: every call below fails a host check first


def kv(**kw):
    base = dict(k=FAKE, v=FAKE, page_table=FAKE, max_pages=8, num_pages=8)
    base.update(kw)
    return _KV(**base)


def draft_call(lib, c, B=1, q=FAKE, k=None, ws=FAKE, ws_bytes=1 << 30, err=FAKE, out=FAKE):
    return lib.seed_draft_attn(ctypes.byref(c), B, q, k or kv(), FAKE, FAKE, FAKE, FAKE, out,
                               None, ws, ws_bytes, err, None)


def test_draft_attn_host_checks(lib):
    c = cfg()
    assert draft_call(lib, c, B=0) == OK                 # empty batch: nothing launched
    assert draft_call(lib, c, B=-1) == ERR_SHAPE
    assert draft_call(lib, c, q=None) == ERR_NULL
    assert draft_call(lib, c, out=None) == ERR_NULL
    assert draft_call(lib, c, err=None) == ERR_NULL
    assert draft_call(lib, c, k=kv(k=None)) == ERR_NULL
    assert draft_call(lib, c, k=kv(max_pages=0)) == ERR_RANGE
    assert draft_call(lib, c, k=kv(num_pages=0)) == ERR_RANGE
    assert draft_call(lib, c, q=FAKE + 8) == ERR_RANGE   # not 16-byte aligned
    assert draft_call(lib, c, ws=FAKE + 128) == ERR_WS   # not 256-byte aligned
    assert draft_call(lib, c, ws_bytes=16) == ERR_WS
    bad = cfg(head_dim=80)
    assert draft_call(lib, bad) == ERR_UNSUP


def test_verify_and_append_host_checks(lib):
    c = cfg()
    assert lib.seed_verify_attn(ctypes.byref(c), 0, FAKE, FAKE, kv(), FAKE, FAKE, None, FAKE,
                                1 << 30, FAKE, None) == OK
    assert lib.seed_verify_attn(ctypes.byref(c), 2, FAKE, None, kv(), FAKE, FAKE, None, FAKE,
                                1 << 30, FAKE, None) == ERR_NULL
    assert lib.seed_verify_attn(ctypes.byref(c), 2, FAKE, FAKE, kv(), FAKE, FAKE, None, FAKE,
                                64, FAKE, None) == ERR_WS
    assert lib.seed_kv_append(ctypes.byref(c), 2, kv(), FAKE, FAKE, None, FAKE, FAKE,
                              None) == ERR_NULL
    assert lib.seed_kv_append(ctypes.byref(c), 2, kv(max_pages=-3), FAKE, FAKE, FAKE, FAKE, FAKE,
                              None) == ERR_RANGE
    assert lib.seed_draft_kv_append(ctypes.byref(c), 2, FAKE, None, FAKE, FAKE, FAKE, FAKE,
                                    None) == ERR_NULL
    assert lib.seed_draft_kv_append(ctypes.byref(c), 0, None, None, None, None, None, None,
                                    None) == OK


def test_accept_host_checks(lib):
    args = [FAKE] * 4 + [8, 16] + [FAKE] * 5
    assert lib.seed_accept_commit(0, 4, *args, None) == OK
    assert lib.seed_accept_commit(2, 0, *args, None) == ERR_SHAPE
    assert lib.seed_accept_commit(2, 32, *args, None) == ERR_SHAPE
    bad = [FAKE, None] + args[2:]
    assert lib.seed_accept_commit(2, 4, *bad, None) == ERR_NULL
    bad = args[:4] + [0, 16] + args[6:]
    assert lib.seed_accept_commit(2, 4, *bad, None) == ERR_RANGE


def test_tree_host_checks(lib):
    c = cfg()
    def tv(cf, B=2, q=FAKE, anc=FAKE, ws_bytes=1 << 30):
        return lib.seed_tree_verify_attn(ctypes.byref(cf), B, q, FAKE, anc, kv(), FAKE, FAKE,
                                         None, FAKE, ws_bytes, FAKE, None)
    assert tv(c, B=0) == OK
    assert tv(c, anc=None) == ERR_NULL
    assert tv(c, q=None) == ERR_NULL
    assert tv(c, ws_bytes=64) == ERR_WS
    # tensor-core kernels only: head_dim 64 takes at most 64 query rows per KV
    # head, head_dim 128 at most 128
    assert tv(cfg(head_dim=64, hq=16, hkv=2, kmax=8)) == ERR_UNSUP   # 8 * 9 rows > 64
    assert tv(cfg(hq=64, hkv=8, kmax=16)) == ERR_UNSUP     # 8 * 17 rows > one 128-row tile
    args = [FAKE] * 5 + [8, 16] + [FAKE] * 6
    assert lib.seed_tree_accept_commit(0, 4, *args, None) == OK
    assert lib.seed_tree_accept_commit(2, 32, *args, None) == ERR_SHAPE
    bad = [FAKE, FAKE, None] + args[3:]
    assert lib.seed_tree_accept_commit(2, 4, *bad, None) == ERR_NULL
    bad = args[:5] + [0, 16] + args[7:]
    assert lib.seed_tree_accept_commit(2, 4, *bad, None) == ERR_RANGE
    assert lib.seed_tree_kv_compact(ctypes.byref(c), 0, kv(), FAKE, FAKE, FAKE, FAKE, None) == OK
    assert lib.seed_tree_kv_compact(ctypes.byref(c), 2, kv(), None, FAKE, FAKE, FAKE,
                                    None) == ERR_NULL
    assert lib.seed_tree_kv_compact(ctypes.byref(c), 2, kv(num_pages=0), FAKE, FAKE, FAKE, FAKE,
                                    None) == ERR_RANGE


def test_draft_head_host_checks(lib):
    args = [FAKE] * 4 + [None, FAKE, 1 << 30, FAKE, None]   # ids..stop, lse, ws, bytes, err, stream
    def call(B=4, d=256, V=1000, h=FAKE, tau=0.7, a=None):
        return lib.seed_draft_head_topk(B, d, V, h, FAKE, ctypes.c_float(tau), *(a or args))
    assert call(B=0) == OK
    assert call(B=129) == ERR_SHAPE
    assert call(d=100) == ERR_SHAPE
    assert call(V=5) == ERR_SHAPE
    assert call(tau=-1.0) == ERR_SHAPE
    assert call(h=None) == ERR_NULL
    assert call(h=FAKE + 8) == ERR_RANGE
    small = args[:6] + [64] + args[7:]
    assert call(a=small) == ERR_WS
    assert lib.seed_draft_head_workspace_bytes(0) == 0
    assert lib.seed_draft_head_workspace_bytes(129) == 0
    assert lib.seed_draft_head_workspace_bytes(64) > 0


def test_linear_host_checks(lib):
    def call(B=4, K=256, N=300, x=FAKE, w=FAKE, w2=None, epi=0, y=FAKE, ws=FAKE, nbytes=1 << 30,
             err=FAKE):
        return lib.seed_linear(B, K, N, x, w, w2, epi, y, ws, nbytes, err, None)
    assert call(B=0) == OK
    assert call(B=129) == ERR_SHAPE
    assert call(K=100) == ERR_SHAPE             # K not a multiple of 64
    assert call(N=0) == ERR_SHAPE
    assert call(epi=3) == ERR_SHAPE
    assert call(x=None) == ERR_NULL
    assert call(epi=2) == ERR_NULL              # SwiGLU needs the up projection
    assert call(w=FAKE + 8) == ERR_RANGE
    assert call(ws=FAKE + 128) == ERR_WS
    assert call(nbytes=64) == ERR_WS
    assert lib.seed_linear_workspace_bytes(4, 300, 100, 0) == 0
    assert lib.seed_linear_workspace_bytes(0, 300, 256, 0) == 0
    a = lib.seed_linear_workspace_bytes(16, 300, 256, 0)
    assert 0 < a < lib.seed_linear_workspace_bytes(16, 300, 256, 2)


def test_draft_layer_host_checks(lib):
    c = _Cfg(32, 8, 128, 16, 8, 0.0)
    P = [FAKE] * 9

    def layer(dm=2560, F=9728, eps=1e-6, theta=1e6):
        return seed._Layer(dm, F, eps, theta, *P)

    def call(cf=c, B=2, L=None, x=FAKE, ws=FAKE, nbytes=1 << 34):
        return lib.seed_draft_layer(ctypes.byref(cf), B, ctypes.byref(L or layer()), x, kv(), FAKE,
                                    FAKE, FAKE, FAKE, ws, nbytes, FAKE, None)
    assert call(B=0) == OK
    assert call(B=129) == ERR_SHAPE
    assert call(L=layer(dm=100)) == ERR_UNSUP
    assert call(L=layer(theta=0.5)) == ERR_UNSUP
    assert call(cf=_Cfg(32, 8, 96, 16, 8, 0.0)) == ERR_UNSUP
    assert call(x=None) == ERR_NULL
    assert call(x=FAKE + 4) == ERR_RANGE
    assert call(nbytes=1024) == ERR_WS
    assert call(ws=FAKE + 16) == ERR_WS
    n = lib.seed_draft_layer_workspace_bytes(ctypes.byref(c), ctypes.byref(layer()), 4)
    assert n > lib.seed_workspace_bytes(ctypes.byref(c), 4)
    assert lib.seed_draft_layer_workspace_bytes(ctypes.byref(c), ctypes.byref(layer()), 0) == 0


def test_block_attn_host_checks(lib):
    c = _Cfg(32, 8, 128, 16, 8, 0.0)

    def call(cf=c, B=2, n=40, b=10, q=FAKE, ws=FAKE, nbytes=1 << 34):
        return lib.seed_block_attn(ctypes.byref(cf), B, n, b, q, FAKE, FAKE, FAKE, FAKE, FAKE,
                                   None, ws, nbytes, FAKE, None)
    assert call(B=0) == OK
    assert call(n=41) == ERR_SHAPE               # n not a multiple of the block
    assert call(b=33, n=66) == ERR_SHAPE         # block above kmax + 1 = 32
    assert call(b=1, n=40) == ERR_SHAPE          # one-token blocks: the draft call's shape
    assert call(cf=_Cfg(32, 8, 96, 16, 8, 0.0)) == ERR_SHAPE
    assert call(q=None) == ERR_NULL
    assert call(q=FAKE + 8) == ERR_RANGE
    # the tensor-core route (head_dim 128, groups 1-4) takes no workspace, so
    # its ws checks are gone (and a valid call would launch: none is made
    # here); the virtual-sequence route still checks it
    c64 = _Cfg(32, 8, 64, 16, 8, 0.0)            # head_dim 64: the virtual-sequence route
    assert call(cf=c64, nbytes=4096) == ERR_WS
    assert call(cf=c64, ws=FAKE + 16) == ERR_WS
    assert call(cf=c64, ws=None) == ERR_NULL
    assert lib.seed_block_attn_workspace_bytes(ctypes.byref(c64), 2, 40, 10) > 4096
    assert lib.seed_block_attn_workspace_bytes(ctypes.byref(c), 2, 40, 10) == 256
    assert lib.seed_block_attn_workspace_bytes(ctypes.byref(c), 2, 41, 10) == 0

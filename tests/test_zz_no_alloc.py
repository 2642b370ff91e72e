"""seed_verify_attn_noalloc, the verify attention that runs on the library's
built-in scratch instead of a caller workspace.

Host side (no GPU): problems whose workspace would not fit the scratch are
refused with SEED_ERR_SCRATCH_LIMIT before any CUDA call, and an invalid cfg
gets the same status as seed_verify_attn.

GPU side: through the C ABI, two calls in a row match seed_verify_attn (with
its own zero-filled workspace) within the parity tolerance, on tensor-core
and CUDA-core shapes with split units, and the second call changes the
device's free memory by nothing.  One shape is also checked against the
oracle (Sec. 4.1 verify attention), and a call whose lengths the kernel
rejects (SEED_DEVERR_CTX_LEN) leaves the scratch fit for the next, valid
call, which again matches the oracle.  The file is named to be collected last, so
that it also runs after every other test in one process.
"""

import ctypes

import numpy as np
import pytest
import torch

from workloads import gen

ATOL, RTOL = 2e-3, 1e-2
SENTINEL = 12345.0
FAKE = 0x10000  # never dereferenced: the calls that use it fail a host check first
DEVERR_CTX_LEN = 1  # SEED_DEVERR_CTX_LEN of include/seed.h


@pytest.fixture(scope="module")
def lib():
    from paper_2609_36590_gb300 import build
    build.build()
    import paper_2609_36590_gb300 as s
    return s.library()


def c_cfg(hq=32, hkv=8, head_dim=128, kmax=8):
    from paper_2609_36590_gb300 import _Cfg
    return _Cfg(hq, hkv, head_dim, 16, kmax, 0.0)


def c_kv():
    from paper_2609_36590_gb300 import _KV
    return _KV(FAKE, FAKE, FAKE, 8, 8)


def test_oversize_problem_is_refused_before_any_cuda_call(lib):
    import paper_2609_36590_gb300 as s
    cfg = c_cfg()
    # the largest batch that fits, and the first one that does not
    fit = max(b for b in range(1, 1024)
              if lib.seed_workspace_bytes(ctypes.byref(cfg), b) <= s.NOALLOC_SCRATCH_BYTES)
    assert fit >= 64   # a 64-sequence, kmax=8 batch of a 32/8-head, D=128 model fits
    st = lib.seed_verify_attn_noalloc(ctypes.byref(cfg), fit + 1, FAKE, FAKE, c_kv(), FAKE,
                                      FAKE, None, FAKE, None)
    assert st == s.SEED_ERR_SCRATCH_LIMIT
    assert b"scratch" in lib.seed_status_string(st)


def test_invalid_cfg_and_empty_batch(lib):
    bad = c_cfg(head_dim=96)
    args = (FAKE, FAKE, c_kv(), FAKE, FAKE, None, FAKE, None)
    assert (lib.seed_verify_attn_noalloc(ctypes.byref(bad), 4, *args)
            == lib.seed_verify_attn(ctypes.byref(bad), 4, FAKE, FAKE, c_kv(), FAKE, FAKE, None,
                                    FAKE, 1 << 20, FAKE, None))
    assert lib.seed_verify_attn_noalloc(ctypes.byref(c_cfg()), 0, *args) == 0
    assert lib.seed_verify_attn_noalloc(None, 4, *args) != 0


# B, hq, hkv, D, kmax, max_ctx: long enough contexts that pairs split into
# several units (the arrival counters in the scratch are used), a D=64 shape
# on the keys-as-rows kernel (20 query rows per KV head), one on the
# CUDA-core kernel (72 rows), the largest kmax, and 12 pairs with a short
# page table (the cluster kernel).
CASES = [
    (6, 32, 8, 128, 4, 3000),
    (5, 32, 8, 128, 8, 1100),
    (4, 16, 16, 128, 16, 700),
    (7, 8, 2, 64, 4, 2500),
    (5, 16, 2, 64, 8, 2500),
    (3, 16, 4, 128, 4, 1500),
]


def dev16(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def paged(rows, nrows, pt, num_pages):
    B, _, hkv, D = rows.shape
    cache = np.full((num_pages, hkv, 16, D), gen.BF16_NAN, dtype=np.uint16)
    for b in range(B):
        pos = np.arange(int(nrows[b]))
        cache[pt[b, pos // 16], :, pos % 16] = rows[b, pos]
    return cache


def assert_close(got, ref, what):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    diff = np.abs(got - ref)
    assert diff.max() <= ATOL, f"{what}: max abs diff {diff.max():.3g}"
    big = np.abs(ref) > 1e-2
    if big.any():
        rel = (diff[big] / np.abs(ref[big])).max()
        assert rel <= RTOL, f"{what}: max rel diff {rel:.3g}"


@pytest.mark.gpu
@pytest.mark.parametrize("case", CASES, ids=lambda c: "B{}_hq{}_hkv{}_D{}_k{}_L{}".format(*c))
def test_noalloc_matches_workspace_entry_point(lib, case):
    assert torch.cuda.is_available(), "GPU test run without a GPU"
    import paper_2609_36590_gb300 as S
    B, hq, hkv, D, kmax, max_ctx = case
    c = gen.small_case(31, B, hq, hkv, D, kmax, max_ctx, True, 1.0)
    cfg = S.SeedConfig(hq=hq, hkv=hkv, head_dim=D, kmax=kmax)
    num_pages = B * c["max_pages"]
    nrows = c["lens"] + c["n_q"]
    kv = S.PagedKV(dev16(paged(c["rows_k"], nrows, c["page_table"], num_pages)),
                   dev16(paged(c["rows_v"], nrows, c["page_table"], num_pages)),
                   torch.from_numpy(c["page_table"]).cuda())
    q = dev16(c["q_verify"])
    n_q = torch.from_numpy(c["n_q"]).cuda()
    lens = torch.from_numpy(c["lens"]).cuda()
    W = kmax + 1

    def outputs():
        return (torch.full((B, W, hq, D), SENTINEL, device="cuda"),
                torch.full((B, W, hq), SENTINEL, device="cuda"),
                torch.zeros(1, dtype=torch.int32, device="cuda"))

    ref_o, ref_l, ref_e = outputs()
    S.seed_verify_attn(cfg, q, n_q, kv, lens, ref_o, ref_l, S.new_workspace(cfg, B), ref_e)

    got = [outputs(), outputs()]
    free = []
    for o, l, e in got:
        S.seed_verify_attn_noalloc(cfg, q, n_q, kv, lens, o, l, e)
        torch.cuda.synchronize()
        free.append(torch.cuda.mem_get_info()[0])
    assert free[0] == free[1], "the second call changed the device's free memory"

    assert int(ref_e.item()) == 0
    ref_o, ref_l = ref_o.cpu().numpy(), ref_l.cpu().numpy()
    for i, (o, l, e) in enumerate(got):
        assert int(e.item()) == 0, f"call {i}: device error {int(e.item())}"
        o, l = o.cpu().numpy(), l.cpu().numpy()
        for b in range(B):
            n = int(c["n_q"][b])
            assert (o[b, n:] == SENTINEL).all() and (l[b, n:] == SENTINEL).all()
            if n:
                assert_close(o[b, :n], ref_o[b, :n], f"call {i} out b={b}")
                assert_close(l[b, :n], ref_l[b, :n], f"call {i} lse b={b}")


def setup_case(S, seed, B, hq, hkv, D, kmax, max_ctx):
    c = gen.small_case(seed, B, hq, hkv, D, kmax, max_ctx, True, 1.0)
    cfg = S.SeedConfig(hq=hq, hkv=hkv, head_dim=D, kmax=kmax)
    num_pages = B * c["max_pages"]
    nrows = c["lens"] + c["n_q"]
    kv = S.PagedKV(dev16(paged(c["rows_k"], nrows, c["page_table"], num_pages)),
                   dev16(paged(c["rows_v"], nrows, c["page_table"], num_pages)),
                   torch.from_numpy(c["page_table"]).cuda())
    return c, cfg, kv


def check_against_oracle(c, o, l, D, what):
    from oracle import attention as OAT
    f64 = gen.bf16_bits_to_f64
    for b in range(len(c["lens"])):
        n, L = int(c["n_q"][b]), int(c["lens"][b])
        assert (o[b, n:] == SENTINEL).all() and (l[b, n:] == SENTINEL).all()
        if n == 0:
            continue
        ro, rl = OAT.verify_attention_seq(f64(c["q_verify"][b, :n]), f64(c["rows_k"][b, :L + n]),
                                          f64(c["rows_v"][b, :L + n]), L, OAT.default_scale(D))
        assert_close(o[b, :n], ro, f"{what} out b={b} L={L} n={n}")
        assert_close(l[b, :n], rl, f"{what} lse b={b}")


@pytest.mark.gpu
def test_noalloc_matches_oracle_and_recovers_after_a_rejected_call(lib):
    assert torch.cuda.is_available(), "GPU test run without a GPU"
    import paper_2609_36590_gb300 as S
    B, hq, hkv, D, kmax, max_ctx = 6, 32, 8, 128, 4, 3000
    c, cfg, kv = setup_case(S, 37, B, hq, hkv, D, kmax, max_ctx)
    q = dev16(c["q_verify"])
    n_q = torch.from_numpy(c["n_q"]).cuda()
    W = kmax + 1

    def call(lens_np):
        o = torch.full((B, W, hq, D), SENTINEL, device="cuda")
        l = torch.full((B, W, hq), SENTINEL, device="cuda")
        e = torch.zeros(1, dtype=torch.int32, device="cuda")
        S.seed_verify_attn_noalloc(cfg, q, n_q, kv, torch.from_numpy(lens_np).cuda(), o, l, e)
        torch.cuda.synchronize()
        return o.cpu().numpy(), l.cpu().numpy(), int(e.item())

    o, l, e = call(c["lens"])
    assert e == 0
    check_against_oracle(c, o, l, D, "noalloc")

    # lengths past the page table's capacity: the kernels' host-independent
    # checks reject those sequences (no row is read for them) and flag it
    bad = c["lens"].copy()
    bad[0] = kv.page_table.shape[1] * 16
    bad[2] = kv.page_table.shape[1] * 16 + 5
    _, _, e = call(bad)
    assert e & DEVERR_CTX_LEN

    o, l, e = call(c["lens"])
    assert e == 0, f"device error {e} after a rejected call"
    check_against_oracle(c, o, l, D, "noalloc after rejected call")

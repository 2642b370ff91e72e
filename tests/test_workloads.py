"""The seeded generators: bf16 rounding, determinism and the planned
acceptance patterns (first mismatch where the plan puts it)."""

import numpy as np
import torch

from workloads import WORKLOADS, gen


def test_bf16_rounding_matches_torch():
    x = np.random.default_rng(0).standard_normal(100000).astype(np.float32) * 7
    x[:5] = [0.0, -0.0, 1.00390625, 1.01171875, 3.0e-39]
    ours = gen.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(ours, ref)
    np.testing.assert_array_equal(gen.bf16_bits_to_f32(ours),
                                  torch.from_numpy(x).to(torch.bfloat16).float().numpy())


def test_blocks_are_deterministic_and_distinct():
    wl = WORKLOADS[2]
    a = gen.ctx_block(wl, 3, 0, 1, gen.K_CTX, 64)
    b = gen.ctx_block(wl, 3, 0, 1, gen.K_CTX, 64)
    c = gen.ctx_block(wl, 3, 0, 2, gen.K_CTX, 64)
    np.testing.assert_array_equal(a, b)
    assert not np.array_equal(a, c)
    v = gen.bf16_bits_to_f64(gen.value_pool(2)[:200000])
    assert abs(v.mean()) < 0.02 and abs(v.std() - 1) < 0.02


def test_key_stress_rows_are_exact_x8():
    wl = WORKLOADS[4]
    n = 4096
    rows = gen.stress_rows(wl, 0, 1, 2, n)
    assert 0.005 < rows.mean() < 0.015
    blk = gen.bf16_bits_to_f64(gen.ctx_block(wl, 0, 1, 2, gen.K_CTX, n))
    raw = gen.bf16_bits_to_f64(gen.window(wl, n * wl.head_dim, gen.K_CTX, 0, 1, 2)).reshape(n, -1)
    np.testing.assert_array_equal(blk[rows], 8 * raw[rows])
    np.testing.assert_array_equal(blk[~rows], raw[~rows])


def test_round_plan_first_mismatch():
    for idx, wl in WORKLOADS.items():
        for rnd in range(min(wl.rounds, 4)):
            k_b, n, draft, target = gen.round_plan(wl, rnd)
            assert (0 <= n).all() and (n <= k_b).all() and (k_b <= wl.kmax).all()
            for b in range(wl.batch):
                eq = draft[b, :k_b[b]] == target[b, :k_b[b]]
                first = int(np.argmin(eq)) if not eq.all() else int(k_b[b])
                assert first == n[b]


def test_page_table_is_a_permutation():
    wl = WORKLOADS[5]
    mp = gen.max_pages(wl)
    pt = gen.page_table(wl, mp)
    assert pt.shape == (wl.batch, mp)
    np.testing.assert_array_equal(np.sort(pt.ravel()), np.arange(wl.batch * mp))
    assert mp * 16 >= gen.ctx_lens(wl).max() + wl.rounds * (wl.kmax + 1)

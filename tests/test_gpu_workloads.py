"""GPU parity on the five synthetic workloads, in the launch configuration the
bench times (one C-ABI call per layer and draft step): the tiny check and the
4B batch-1 shape in full; batch 16, the 32k-token stress case and the 32-round
paged serving mix on sampled layers and sequences, computed one by one by the
oracle; in the serving mix, every rolled-back cache slot is overwritten with
NaN after each accept, so a read of one would show as a non-finite output.  Accepted lengths, tokens, committed slots and lengths: bit-exact every
round.  Attention: max abs <= 2e-3, max rel <= 1e-2 (|o| > 1e-2)."""

import numpy as np
import pytest
import torch

from oracle.workload import OracleRun
from workloads import WORKLOADS

pytestmark = pytest.mark.gpu

ATOL, RTOL = 2e-3, 1e-2


def assert_close(got, ref, what):
    got = np.asarray(got, dtype=np.float64)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    diff = np.abs(got - ref)
    assert diff.max() <= ATOL, f"{what}: max abs err {diff.max():.3g}"
    big = np.abs(ref) > 1e-2
    if big.any():
        rel = (diff[big] / np.abs(ref[big])).max()
        assert rel <= RTOL, f"{what}: max rel err {rel:.3g}"


@pytest.fixture(scope="module")
def DW():
    assert torch.cuda.is_available(), "GPU test run without a GPU"
    from paper_2609_36590_gb300 import build
    build.build()
    from workloads.device import DeviceWorkload
    return DeviceWorkload


def poison_rolled_back(dw, lens_before, k_b):
    """Write bf16 NaN into every cache slot that the round's verify appended
    and the accept rolled back (positions L + n + 1 .. L + k_b of each
    sequence, in every materialised layer), so that any later read of a
    rolled-back row would turn that output into NaN (Alg. 2: only the
    accepted prefix is committed)."""
    acc = dw.accepted.cpu().numpy()
    n = 0
    for b in range(len(lens_before)):
        lo, hi = int(lens_before[b]) + int(acc[b]) + 1, int(lens_before[b]) + int(k_b[b])
        if hi < lo:
            continue
        pos = np.arange(lo, hi + 1)
        pages = torch.from_numpy(dw.pt_np[b, pos // 16].astype(np.int64)).to(dw.device)
        slots = torch.from_numpy((pos % 16).astype(np.int64)).to(dw.device)
        for l in dw.layers:
            dw.kv[l].k[pages, :, slots] = float("nan")
            dw.kv[l].v[pages, :, slots] = float("nan")
        n += len(pos)
    return n


def run_and_check(DW, idx, layers=None, rounds=None, sample_b=None, verify_layers=None,
                  poison=False):
    """Run the workload's rounds on the GPU; check every accept bit-exactly and
    the attention outputs of the sampled (layer, sequence) pairs.  poison:
    after every accept, NaN into the rolled-back slots (poison_rolled_back)."""
    wl = WORKLOADS[idx]
    n_rounds = wl.rounds if rounds is None else rounds
    dw = DW(wl, layers=layers, rounds=n_rounds)
    orc = OracleRun(wl, rounds=n_rounds)
    np.testing.assert_array_equal(orc.page_table, dw.pt_np)
    checked = poisoned = 0
    for rnd in range(n_rounds):
        bs = list(range(wl.batch)) if sample_b is None else sample_b(rnd)
        vl = dw.layers if verify_layers is None else verify_layers(rnd)
        got_d, got_v = {}, {}

        def on_draft(i, l, out, lse):
            got_d[(i, l)] = (out[bs].cpu().numpy(), lse[bs].cpu().numpy())

        def on_verify(l, out, lse):
            if l in vl:
                got_v[l] = (out[bs].cpu().numpy(), lse[bs].cpu().numpy())

        lens_before = dw.ctx_lens.cpu().numpy().copy()
        dw.run_round(rnd, on_draft=on_draft, on_verify=on_verify)
        torch.cuda.synchronize()
        assert int(dw.err.item()) == 0, f"device error flag {int(dw.err.item())}"

        for (i, l), (o_g, l_g) in got_d.items():
            ref = orc.draft(rnd, i, l, bs)
            for k, b in enumerate(bs):
                if b in ref:
                    assert_close(o_g[k], ref[b][0], f"wl{idx} r{rnd} draft step {i} layer {l} b{b}")
                    assert_close(l_g[k], ref[b][1], f"wl{idx} r{rnd} draft lse {i} {l} b{b}")
                    checked += 1
        for l, (o_g, l_g) in got_v.items():
            ref = orc.verify(rnd, l, bs)
            for k, b in enumerate(bs):
                n = ref[b][0].shape[0]
                assert_close(o_g[k, :n], ref[b][0], f"wl{idx} r{rnd} verify layer {l} b{b}")
                assert_close(l_g[k, :n], ref[b][1], f"wl{idx} r{rnd} verify lse {l} b{b}")
                checked += 1

        acc, tok, slots, new_lens = orc.accept(rnd)
        np.testing.assert_array_equal(dw.accepted.cpu().numpy(), acc)
        np.testing.assert_array_equal(dw.tokens.cpu().numpy(), tok)
        np.testing.assert_array_equal(dw.slots.cpu().numpy(), slots)
        np.testing.assert_array_equal(dw.ctx_lens.cpu().numpy(), new_lens)
        if poison:
            poisoned += poison_rolled_back(dw, lens_before, dw.round_inputs(rnd)["k_b_np"])
        orc._ctx_cache.clear()
    assert checked > 0
    assert poisoned > 0 or not poison
    return dw, orc


def test_workload1_tiny_full(DW):
    run_and_check(DW, 1)


def test_workload2_4b_batch1_all_layers(DW):
    run_and_check(DW, 2)


def test_workload3_batch16_sampled_layers(DW):
    run_and_check(DW, 3, layers=[0, 13, 26, 27])


def test_workload4_long_context_sampled(DW):
    run_and_check(DW, 4, layers=[5, 26, 27], sample_b=lambda r: [0, 3])


def test_workload5_serving_mix_32_rounds(DW):
    wl = WORKLOADS[5]
    rng = np.random.default_rng(5)
    picks = [sorted(rng.choice(wl.batch, size=3, replace=False).tolist()) for _ in range(wl.rounds)]
    layers = [3, 11, 26, 27]
    dw, orc = run_and_check(DW, 5, layers=layers, sample_b=lambda r: picks[r],
                            verify_layers=lambda r: [layers[r % 2], 26, 27], poison=True)
    assert (orc.lens > orc.lens0).all()

"""The five synthetic workloads of the draft/verify attention path.

Each workload is shaped like the paper's 4B-scale decode (Sec. 4.1: a 28-layer
decoder split into a 26-layer encoder and a 2-layer decoder; Appendix, cost
analysis: 8 KV heads of width 128) or, for the tiny check, a one-layer model.
The paper measures on GSM8K / KodCode / ScienceQA / CNN-DM; none of that data
is used or needed here: every tensor is drawn from the seeded generators in
``workloads.gen``.
"""

from __future__ import annotations

from dataclasses import dataclass


PAGE_SIZE = 16  # tokens per KV-cache page


@dataclass(frozen=True)
class Workload:
    index: int            # 1..5
    name: str
    n_layers: int         # layers whose attention runs in one verify step
    dec_layers: tuple     # 0-based layers the drafter (f_dec) runs
    hq: int
    hkv: int
    head_dim: int
    batch: int
    kmax: int             # maximum draft length d
    rounds: int           # consecutive draft-verify rounds in the workload
    ctx: str              # 'fixed' | 'uniform' | 'loguniform'
    ctx_lo: int
    ctx_hi: int
    accept: str           # 'forced' | 'uniform' | 'geom'
    ragged_k: bool        # per-sequence draft length drawn each round
    key_stress: float     # fraction of key rows scaled by 8
    paged_random: bool    # pages in a seeded random order (else identity)
    vocab: int = 1000
    geom_p: float = 0.3

    @property
    def group(self) -> int:
        return self.hq // self.hkv

    @property
    def row_bytes(self) -> int:
        """K+V bytes of one token in one layer (bf16)."""
        return 2 * self.hkv * self.head_dim * 2


WORKLOADS = {
    1: Workload(1, "tiny-1L-8q2kv-d64-b1-L256-k4", n_layers=1, dec_layers=(0,),
                hq=8, hkv=2, head_dim=64, batch=1, kmax=4, rounds=1,
                ctx="fixed", ctx_lo=256, ctx_hi=256, accept="forced",
                ragged_k=False, key_stress=0.0, paged_random=False),
    2: Workload(2, "4B-28L-32q8kv-d128-b1-L2048-k4", n_layers=28, dec_layers=(26, 27),
                hq=32, hkv=8, head_dim=128, batch=1, kmax=4, rounds=1,
                ctx="fixed", ctx_lo=2048, ctx_hi=2048, accept="uniform",
                ragged_k=False, key_stress=0.0, paged_random=False),
    3: Workload(3, "4B-28L-32q8kv-d128-b16-L1024..4096-k4", n_layers=28, dec_layers=(26, 27),
                hq=32, hkv=8, head_dim=128, batch=16, kmax=4, rounds=1,
                ctx="uniform", ctx_lo=1024, ctx_hi=4096, accept="geom",
                ragged_k=False, key_stress=0.0, paged_random=False),
    4: Workload(4, "4B-28L-32q8kv-d128-b4-L32768-k8-keyx8", n_layers=28, dec_layers=(26, 27),
                hq=32, hkv=8, head_dim=128, batch=4, kmax=8, rounds=1,
                ctx="fixed", ctx_lo=32768, ctx_hi=32768, accept="geom",
                ragged_k=False, key_stress=0.01, paged_random=False),
    5: Workload(5, "4B-28L-32q8kv-d128-b64-L512..8192-paged16-k1..8-32rounds", n_layers=28,
                dec_layers=(26, 27), hq=32, hkv=8, head_dim=128, batch=64, kmax=8, rounds=32,
                ctx="loguniform", ctx_lo=512, ctx_hi=8192, accept="uniform",
                ragged_k=True, key_stress=0.0, paged_random=True),
}


def get(index: int) -> Workload:
    return WORKLOADS[int(index)]

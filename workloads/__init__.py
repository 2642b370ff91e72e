"""Seeded synthetic workloads for the SEED draft/verify attention path.

Holds workload definitions (``configs``) and the seeded input generators
(``gen``).  Nothing here computes attention or acceptance; both the CUDA path
and the oracle draw their inputs from here.
"""

from .configs import PAGE_SIZE, WORKLOADS, Workload, get  # noqa: F401

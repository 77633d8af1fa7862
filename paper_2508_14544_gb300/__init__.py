"""GB300-native batched simulator of the schedulers of arXiv 2508.14544 (A_max, A_min, H-SF, and the
auxiliary A_r and promote-l A_ell policies).

The simulation runs in hand-written CUDA kernels behind the C ABI of ``include/sim.h``
(``libsim.so``); this package holds the build step, the ctypes binding and the seeded
synthetic workload generator.
"""
from ._lib import (SIM_AMAX, SIM_AMIN, SIM_HSF, SIM_AR, SIM_AELL, RESULT_DTYPE, SimError, lib, sim_create, sim_load,
                   sim_load_csr, sim_load_ranked_csr, sim_run, sim_get_completions, sim_competitive_ratio, sim_set_option, sim_last_error, sim_destroy,
                   sim_kernel_launches, cr_amin_lemma, cr_amin_rho)
from .sim import Simulator

POLICIES = {"A_max": SIM_AMAX, "A_min": SIM_AMIN, "H-SF": SIM_HSF, "A_r": SIM_AR, "A_ell": SIM_AELL}

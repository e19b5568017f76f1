"""A pin of the oracle's Philox4x32-10 that does not depend on stored
values: cuRAND's device generator of the same name, run through its public
API (curand_init with a seed, a subsequence and an offset, then curand4),
must give the same 128-bit blocks for counters whose four words are all in
use (offset / 4 in words 0-1, the subsequence in words 2-3) and keys of
every kind.  The probe, tests/curand_philox_probe.cu, is compiled by the
package's build step (with the nvcc that builds libedp) or here, the same
way, when that step has not made it."""
import ctypes as C

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def probe():
    from paper_2609_24456_gb300 import build
    lib = C.CDLL(build.build_curand_probe())
    lib.curand_philox_probe.argtypes = [C.c_void_p] * 3 + [C.c_uint, C.c_void_p]
    lib.curand_philox_probe.restype = C.c_int
    return lib


def test_oracle_philox_matches_curand(probe, orc):
    rng = np.random.default_rng(2024)
    n = 4096
    seed = rng.integers(0, 2**64, size=n, dtype=np.uint64)
    seed[:4] = [0, 2**64 - 1, 0x0123456789ABCDEF, 1]
    sub = rng.integers(0, 2**64, size=n, dtype=np.uint64)
    sub[:4] = [0, 2**64 - 1, 7, 2**32]
    j = rng.integers(0, 2**62, size=n, dtype=np.uint64)
    j[:4] = [0, 2**62 - 1, 77, 2**32 + 5]
    off = j * np.uint64(4)
    dev = lambda a: torch.from_numpy(a.view(np.int64)).cuda()
    d_seed, d_sub, d_off = dev(seed), dev(sub), dev(off)
    out = torch.zeros((n, 4), dtype=torch.int32, device="cuda")
    assert probe.curand_philox_probe(d_seed.data_ptr(), d_sub.data_ptr(), d_off.data_ptr(),
                                     n, out.data_ptr()) == 0
    got = out.cpu().numpy().view(np.uint32)
    M = 0xFFFFFFFF
    for i in range(n):
        s, q, jj = int(seed[i]), int(sub[i]), int(j[i])
        ref = orc.philox4x32_10([jj & M, jj >> 32, q & M, q >> 32], [s & M, s >> 32])
        assert list(got[i]) == [int(x) for x in ref], i

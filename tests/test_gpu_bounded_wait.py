"""The bounded mbarrier wait of the staged frame-stack delivery expires
instead of hanging.  The probe (tests/mbar_wait_probe.cu, built by the
package's build step) runs libedp's wait helper on an mbarrier that nothing
arrives on: the wait must return false after about its limit (here 2 ms),
with the GPU context still usable; after the thread's own arrival the same
wait returns true at once.  The delivery kernel uses the same helper (with a
1 s limit) and reports an expiry as DEVERR_TIMEOUT."""
import ctypes as C

import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def probe():
    from paper_2609_24456_gb300 import build
    lib = C.CDLL(build.build_wait_probe())
    lib.mbar_wait_probe.argtypes = [C.c_uint64, C.c_void_p]
    lib.mbar_wait_probe.restype = C.c_int
    return lib


def test_wait_expires_and_context_stays_usable(probe):
    out = torch.zeros(4, dtype=torch.int64, device="cuda")
    limit = 2_000_000  # ns
    assert probe.mbar_wait_probe(limit, out.data_ptr()) == 0
    got, waited, got2, waited2 = out.tolist()
    assert got == 0, "a wait with no arrival must expire"
    assert limit <= waited < 1_000_000_000
    assert got2 == 1 and waited2 < limit
    # the context still runs work
    x = torch.arange(1024, device="cuda", dtype=torch.float32)
    assert float(x.sum()) == 1023 * 1024 / 2

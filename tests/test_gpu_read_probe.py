"""The read probe (aq_selftest_read) that the benchmark uses as the per-call floor of reading a
GEMV's code bytes: it must read every byte exactly once, which the XOR fold of all 32-bit words
shows (compared with numpy's fold of the same bytes), over sizes with and without a partial
last kilobyte, with fewer chunks than SMs and with several chunks per warp."""
import numpy as np
import pytest
import torch

import aq_testutil as U
import paper_2606_12876_gb300 as aq

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    U.require_gpu()


@pytest.mark.parametrize("nbytes", [0, 16, 1024, 1040, 152 * 1024, 3 * 152 * 1024 + 528,
                                    (8 << 20) + 48, 29360128])
def test_read_probe_folds_every_word(nbytes):
    rng = np.random.default_rng(nbytes)
    host = rng.integers(0, 2**32, size=(nbytes + 64) // 4, dtype=np.uint32)
    src = torch.from_numpy(host.view(np.int32)).cuda()
    sink = torch.zeros(4, dtype=torch.int32, device="cuda")
    aq.aq_selftest_read(src, nbytes, sink)
    got = int(sink[0].item()) & 0xffffffff
    want = int(np.bitwise_xor.reduce(host[: nbytes // 4])) if nbytes else 0
    assert got == want

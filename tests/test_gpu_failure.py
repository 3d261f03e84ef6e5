"""The failure path of the bounded waits on the GPU, without a fault.

Every wait of the product kernels on an mbarrier is bounded; when one expires the kernel sets
FQT1_DEV_TIMEOUT in the caller's status word, lets its in-flight copies land, frees its tensor
memory and returns.  fqt1_test_expired_wait runs the forward product's kernel with one arrive
withheld (a flag nothing sets), so its wait runs out after 20 ms.  The test checks the status
bit, that the launch returned normally, and that the same context then computes a correct
product.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

from oracle import method as om  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2408_14267_gb300 import build
    build.build()


def test_expired_wait_sets_status_and_context_survives():
    from paper_2408_14267_gb300 import fqt1
    rng = np.random.default_rng(5)
    M, K, D = 384, 2304, 256
    a = rng.standard_normal((M, K)).astype(np.float32)
    b = rng.standard_normal((D, K)).astype(np.float32)
    dev = torch.device("cuda")
    wK = fqt1.packed_words(K)
    sa = torch.empty(M, wK, dtype=torch.int32, device=dev)
    sb = torch.empty(D, wK, dtype=torch.int32, device=dev)
    fqt1.binarize_pack(torch.from_numpy(a).cuda(), M, K, K, sa, None, None)
    fqt1.binarize_pack(torch.from_numpy(b).cuda(), D, K, K, sb, None, None)
    gamma = torch.ones(D, device=dev)
    y = torch.empty(M, D, device=dev)
    status = torch.zeros(4, dtype=torch.int32, device=dev)
    fqt1.test_expired_wait(sa, sb, M, D, K, gamma, y, status)
    torch.cuda.synchronize()  # raises if the kernel faulted
    assert int(status[0].item()) & 0x200, "the withheld arrive must expire a bounded wait"
    # the context is still usable: a normal product right after is exact
    acc = torch.empty(M, D, dtype=torch.int32, device=dev)
    fqt1.fwd_gemm(sa, sb, M, D, K, gamma, acc, y)
    torch.cuda.synchronize()
    assert np.array_equal(acc.cpu().numpy(), om.int_matmul(om.sign(a), om.sign(b)))

"""Eq. 10 importance scores on the GPU (qsvd_importance_scores) against
oracle.rank (itself pinned to Eq. 9's definition).  fp32 with atomic
accumulation: relative tolerance 1e-4 of the largest score."""
import numpy as np
import pytest
import torch

from gpu_util import dev, q
from oracle import rank

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("N,m,n,k", [(1, 64, 32, 64), (3, 200, 150, 70), (2, 96, 300, 129)])
def test_importance_scores_match_oracle(N, m, n, k):
    """Tiles of 64 singular values and 64 rows with ragged edges; k > n and
    k < n."""
    rng = np.random.default_rng(N * 1000 + m)
    U = rng.standard_normal((m, k)) / np.sqrt(m)
    s = np.sort(rng.uniform(0.1, 3.0, k))[::-1].copy()
    Vt = rng.standard_normal((k, n)) / np.sqrt(n)
    G = rng.standard_normal((N, m, n))
    f = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev())  # noqa: E731
    got = q().qsvd_importance_scores(f(U), f(s), f(Vt), f(G)).cpu().numpy().astype(np.float64)
    q().qsvd_check()
    # the oracle on the same fp32-rounded inputs
    r32 = lambda a: np.asarray(a, dtype=np.float32).astype(np.float64)  # noqa: E731
    want = rank.importance_scores(r32(U), r32(s), r32(Vt), [r32(g) for g in G])
    np.testing.assert_allclose(got, want, rtol=1e-4, atol=1e-4 * want.max())


def test_importance_argument_errors():
    lib = q()
    z = torch.zeros((4, 4), dtype=torch.float32, device=dev())
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_importance_scores(z, torch.zeros(4, device=dev()), z, torch.zeros((1, 4, 4), device=dev()),
                                   workspace=torch.zeros(4, dtype=torch.uint8, device=dev()))
    assert e.value.status == lib.QSVD_ENOSPC

"""The allocation-free projection entry point (dllm_op_gemm_noalloc).

Some callers cannot allocate device memory: code running while a stream is
captured into a CUDA graph, or an application whose device memory belongs to
its own pool.  For them the library offers a variant of the tensor-core
projection whose scratch sits in a static device array.  This checks, through
the C ABI, that it returns what the allocating entry point (dllm_op_gemm)
returns, within the tolerance of the GEMM tests, on two calls in a row (the
second call reuses the array the first one left behind).  The file is named so
that pytest collects it last.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("M,N,K", [(4096, 32, 4096), (200, 40, 688), (1024, 96, 1024)])
def test_noalloc_gemm_matches_allocating_entry_point(M, N, K):
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2606_13740_gb300 import dllm
    dllm.lib()
    dev = torch.device("cuda:0")
    rng = np.random.default_rng(M + N + K)
    W = torch.from_numpy((rng.standard_normal((M, K)) * 0.05).astype(np.float32)).to(torch.bfloat16).to(dev)
    X = torch.from_numpy(rng.standard_normal((N, K)).astype(np.float32)).to(torch.bfloat16).to(dev)
    ref = dllm.dllm_op_gemm(W, X, M, N, K).cpu().numpy()
    w64 = W.float().cpu().numpy().astype(np.float64)
    x64 = X.float().cpu().numpy().astype(np.float64)
    scale = np.sqrt((x64 ** 2).sum(1))[:, None] * np.sqrt((w64 ** 2).sum(1))[None, :]
    for _ in range(2):
        D = torch.full((N, M), float("nan"), dtype=torch.float32, device=dev)
        dllm.dllm_op_gemm_noalloc(W, X, D, M, N, K)
        got = D.cpu().numpy()
        assert np.all(np.abs(got - ref) <= 1e-5 * scale + 1e-6), np.abs(got - ref).max()


def test_noalloc_gemm_rejects_oversized_grid():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2606_13740_gb300 import dllm
    dev = torch.device("cuda:0")
    M, N, K = 4096, 256, 4096  # 2048 k-block iterations, 256 KiB of partials per CTA
    W = torch.zeros((M, K), dtype=torch.bfloat16, device=dev)
    X = torch.zeros((N, K), dtype=torch.bfloat16, device=dev)
    D = torch.empty((N, M), dtype=torch.float32, device=dev)
    with pytest.raises(dllm.DllmError) as e:
        dllm.dllm_op_gemm_noalloc(W, X, D, M, N, K, grid=2048)
    assert e.value.code == -6

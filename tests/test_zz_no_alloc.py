"""The allocation-free projection entry point (dllm_op_gemm_noalloc).

Some callers cannot allocate device memory: an application that hands nearly
all of a GPU's memory to its own pool allocator (a library's cudaMalloc then
fails or breaks its accounting), or a latency-critical loop that cannot take
the implicit synchronisation of cudaMalloc and cudaFree.  For them the library
offers a variant of the tensor-core projection whose scratch sits in one static
device array.  These tests call it through the C ABI and check, on two calls in
a row (the second reuses the array the first left behind), that it returns what
the allocating entry point (dllm_op_gemm) returns and what an fp64 product of
the same bf16 operands gives, within the tolerance of the GEMM tests; that an
automatically chosen grid shrinks to fit the array; and that sizes beyond its
limits are rejected.  The file is named so that pytest collects it last.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dllm():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2606_13740_gb300 import dllm as d
    d.lib()
    return d


def _operands(M, N, K):
    rng = np.random.default_rng(M + N + K)
    dev = torch.device("cuda:0")
    W = torch.from_numpy((rng.standard_normal((M, K)) * 0.05).astype(np.float32)).to(torch.bfloat16).to(dev)
    X = torch.from_numpy(rng.standard_normal((N, K)).astype(np.float32)).to(torch.bfloat16).to(dev)
    return W, X


# (4096, 256, 4096): 256-token tiles, 128 KiB of partials per CTA, so the automatic grid shrinks
# from one CTA per SM to the 62 CTAs whose partials fit the static array
@pytest.mark.parametrize("M,N,K", [(4096, 32, 4096), (200, 40, 688), (1024, 96, 1024), (4096, 256, 4096)])
def test_noalloc_gemm_matches_allocating_entry_point(dllm, M, N, K):
    W, X = _operands(M, N, K)
    ref = dllm.dllm_op_gemm(W, X, M, N, K).cpu().numpy()
    w64 = W.float().cpu().numpy().astype(np.float64)
    x64 = X.float().cpu().numpy().astype(np.float64)
    exact = x64 @ w64.T
    scale = np.sqrt((x64 ** 2).sum(1))[:, None] * np.sqrt((w64 ** 2).sum(1))[None, :]
    tol = 1e-5 * scale + 1e-6
    assert np.all(np.abs(ref - exact) <= tol)
    for _ in range(2):
        D = torch.full((N, M), float("nan"), dtype=torch.float32, device=W.device)
        dllm.dllm_op_gemm_noalloc(W, X, D, M, N, K)
        got = D.cpu().numpy()
        assert np.all(np.abs(got - exact) <= tol), np.abs(got - exact).max()
        assert np.all(np.abs(got - ref) <= tol), np.abs(got - ref).max()


def test_noalloc_gemm_rejects_oversized_grid(dllm):
    dev = torch.device("cuda:0")
    M, N, K = 4096, 256, 4096  # 128 KiB of partials per CTA: at most 62 CTAs fit
    W = torch.zeros((M, K), dtype=torch.bfloat16, device=dev)
    X = torch.zeros((N, K), dtype=torch.bfloat16, device=dev)
    D = torch.empty((N, M), dtype=torch.float32, device=dev)
    with pytest.raises(dllm.DllmError) as e:
        dllm.dllm_op_gemm_noalloc(W, X, D, M, N, K, grid=100)
    assert e.value.code == -6


def test_noalloc_gemm_rejects_too_many_tiles(dllm):
    dev = torch.device("cuda:0")
    M, N, K = 128 * 2047, 32, 64  # 2047 output tiles, one more than the array's tickets
    W = torch.zeros((M, K), dtype=torch.bfloat16, device=dev)
    X = torch.zeros((N, K), dtype=torch.bfloat16, device=dev)
    D = torch.empty((N, M), dtype=torch.float32, device=dev)
    with pytest.raises(dllm.DllmError) as e:
        dllm.dllm_op_gemm_noalloc(W, X, D, M, N, K)
    assert e.value.code == -6

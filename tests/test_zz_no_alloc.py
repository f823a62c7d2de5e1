"""gs_linear_noalloc: the projection GEMM for callers that cannot allocate
device memory (an operator with no workspace argument, a plugin host whose
allocator owns the device memory, a real-time path that must not trigger
cudaMalloc's synchronisation).  Its split-K scratch lives in a fixed device
array inside the library; this checks it against gs_linear, which takes the
same scratch from the caller, on two calls in a row through the C ABI.

Kept in a file of its own that pytest collects last.
"""
import pytest
import torch

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def gs():
    from paper_2609_26638_gb300 import gs as binding
    return binding


def _with_caller_scratch(gs, x, w, M, N, K, epi, split, y):
    sb = gs.gs_linear_scratch_bytes(M, N, split)
    scratch = torch.zeros(sb, dtype=torch.uint8, device=DEV)
    gs.gs_linear(x.data_ptr(), w.data_ptr(), y.data_ptr(), M, N, K, epi, split, scratch.data_ptr(),
                 sb, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()


def test_noalloc_matches_linear_on_two_calls_in_a_row(gs):
    stream = torch.cuda.current_stream().cuda_stream
    g = torch.Generator(device=DEV).manual_seed(11)
    cases = [(17, 2048, 1024, gs.EPI_STORE_F16, 8), (9, 1024, 4096, gs.EPI_STORE_F16, 16)]
    for M, N, K, epi, split in cases:          # two calls in a row share the one array
        x = torch.randn(M, K, device=DEV, generator=g).half()
        w = (0.02 * torch.randn(N, K, device=DEV, generator=g)).half()
        want = torch.zeros(M, N, dtype=torch.float16, device=DEV)
        _with_caller_scratch(gs, x, w, M, N, K, epi, split, want)
        got = torch.zeros(M, N, dtype=torch.float16, device=DEV)
        gs.gs_linear_noalloc(x.data_ptr(), w.data_ptr(), got.data_ptr(), M, N, K, epi, split, stream)
        assert gs.gs_linear_noalloc_status(stream) == gs.GS_OK     # synchronises the stream
        ref = x.float() @ w.float().T
        torch.testing.assert_close(got.float(), want.float(), rtol=1e-2,
                                   atol=1e-2 * ref.abs().max().item())
        torch.testing.assert_close(got.float(), ref, rtol=1e-2, atol=1e-2 * ref.abs().max().item())


@pytest.mark.parametrize("M,N,K,epi,split", [
    (17, 1024, 4096, 1, 8),       # residual add; gs_linear reduces its splits in a cluster
    (200, 1024, 1024, 1, 2),      # 256-token tile here, 64-token cluster tiles in gs_linear
    (72, 512, 1024, 2, 4),        # SwiGLU; gs_linear sums the four chunks inside one CTA
    (100, 4096, 1024, 3, 2),      # LM-head argmax keys
    (300, 2048, 1024, 0, 1),      # no split: two 256-token tiles
])
def test_noalloc_equals_linear_bitwise(gs, M, N, K, epi, split):
    """Same split-K factor, so the same K chunks summed in the same order:
    whatever tile width or reduction path each entry point takes, the
    outputs are identical bit for bit, and the kernel-side status is clean."""
    stream = torch.cuda.current_stream().cuda_stream
    g = torch.Generator(device=DEV).manual_seed(M * 31 + epi)
    wrows = 2 * N if epi == gs.EPI_SWIGLU else N
    x = torch.randn(M, K, device=DEV, generator=g).half()
    w = (0.02 * torch.randn(wrows, K, device=DEV, generator=g)).half()
    if epi == gs.EPI_RESID_F32:
        base = torch.randn(M, N, device=DEV, generator=g)
        want, got = base.clone(), base.clone()
    elif epi == gs.EPI_ARGMAX:
        want = torch.zeros(M, dtype=torch.int64, device=DEV)
        got = torch.zeros(M, dtype=torch.int64, device=DEV)
    else:
        want = torch.zeros(M, N, dtype=torch.float16, device=DEV)
        got = torch.zeros(M, N, dtype=torch.float16, device=DEV)
    _with_caller_scratch(gs, x, w, M, N, K, epi, split, want)
    gs.gs_linear_noalloc(x.data_ptr(), w.data_ptr(), got.data_ptr(), M, N, K, epi, split, stream)
    assert gs.gs_linear_noalloc_status(stream) == gs.GS_OK
    assert torch.equal(got, want)


def test_noalloc_rejects_scratch_beyond_its_array(gs):
    # 64 k-block splits over 64 feature tiles of 32 rows need 64 MiB of partials > 8 MiB
    x = torch.zeros(17, 4096, dtype=torch.float16, device=DEV)
    w = torch.zeros(8192, 4096, dtype=torch.float16, device=DEV)
    y = torch.zeros(17, 8192, dtype=torch.float16, device=DEV)
    with pytest.raises(gs.GsError) as e:
        gs.gs_linear_noalloc(x.data_ptr(), w.data_ptr(), y.data_ptr(), 17, 8192, 4096,
                             gs.EPI_STORE_F16, 64, torch.cuda.current_stream().cuda_stream)
    assert e.value.code == gs.GS_ERR_OOM


def test_noalloc_status_reports_a_range_overflow_then_clears(gs):
    """Outputs beyond the fp16 range set the private error word; the status
    query reports it once (GS_ERR_DEVICE_CHECK) and clears it."""
    stream = torch.cuda.current_stream().cuda_stream
    x = torch.full((17, 1024), 256.0, dtype=torch.float16, device=DEV)
    w = torch.full((256, 1024), 256.0, dtype=torch.float16, device=DEV)
    y = torch.zeros(17, 256, dtype=torch.float16, device=DEV)
    gs.gs_linear_noalloc(x.data_ptr(), w.data_ptr(), y.data_ptr(), 17, 256, 1024,
                         gs.EPI_STORE_F16, 1, stream)
    assert gs.gs_linear_noalloc_status(stream) == gs.GS_ERR_DEVICE_CHECK
    assert gs.gs_linear_noalloc_status(stream) == gs.GS_OK
    x.fill_(1.0 / 64)
    gs.gs_linear_noalloc(x.data_ptr(), w.data_ptr(), y.data_ptr(), 17, 256, 1024,
                         gs.EPI_STORE_F16, 1, stream)
    assert gs.gs_linear_noalloc_status(stream) == gs.GS_OK
    assert torch.all(y == 4096.0)                       # 1024 * 256 / 64, exact in fp16

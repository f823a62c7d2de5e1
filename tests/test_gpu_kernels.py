"""Kernel-level GPU parity: the tcgen05 GEMM against a plain fp32 torch matmul
of the same fp16 operands, and the paged hybrid-mask attention against the
oracle's float64 masked softmax (draft and verify masks from the oracle's mask
builders).

Tolerances follow from the arithmetic: products are exact in fp32 and
accumulate in fp32 (relative error ~K * 2^-24), so a GEMM output carries the
fp16 rounding of its store, 2^-11 relative; attention carries the fp16
rounding of the probabilities fed to P.V (each p within 2^-11 relative, so
the output within 2^-11 * max|v|) plus the fp16 store of the output."""
import math
import types

import numpy as np
import pytest
import torch

import synth
from oracle import decode as od
from oracle.model import Decoder

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def gs():
    from paper_2609_26638_gb300 import gs as binding
    return binding


def _linear(gs, x, w, M, N, K, epi, split, y):
    sb = gs.gs_linear_scratch_bytes(M, N, split)
    scratch = torch.zeros(sb, dtype=torch.uint8, device=DEV)
    gs.gs_linear(x.data_ptr(), w.data_ptr(), y.data_ptr(), M, N, K, epi, split, scratch.data_ptr(),
                 sb, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()


@pytest.mark.parametrize("M", [1, 17, 33, 100, 264, 544])
@pytest.mark.parametrize("N,K,split", [(256, 256, 1), (2048, 1024, 8), (1024, 4096, 16),
                                       (1024, 4096, 32)])
def test_linear_store_and_residual(gs, M, N, K, split):
    g = torch.Generator(device=DEV).manual_seed(M * 7 + N)
    x = torch.randn(M, K, device=DEV, generator=g).half()
    w = (0.02 * torch.randn(N, K, device=DEV, generator=g)).half()
    ref = x.float() @ w.float().T
    y = torch.zeros(M, N, dtype=torch.float16, device=DEV)
    _linear(gs, x, w, M, N, K, gs.EPI_STORE_F16, split, y)
    torch.testing.assert_close(y.float(), ref, rtol=2e-3, atol=1e-3 * ref.abs().max().item())
    base = torch.randn(M, N, device=DEV, generator=g)
    r = base.clone()
    _linear(gs, x, w, M, N, K, gs.EPI_RESID_F32, split, r)
    torch.testing.assert_close(r, base + ref, rtol=1e-4, atol=1e-4 * ref.abs().max().item())


@pytest.mark.parametrize("M,N,K,split", [(9, 1024, 4096, 16), (100, 1024, 4096, 32)])
def test_linear_clears_stale_scratch(gs, M, N, K, split):
    """Split-K through global scratch (no cluster, no in-CTA chunks): the
    caller's scratch arrives full of stale bytes (0x7f), as from a caching
    allocator; the call clears the arrival counters and the error word itself,
    so every tile is written once from all its partial sums, and the error
    word (first int32) reads 0 afterwards."""
    g = torch.Generator(device=DEV).manual_seed(M + split)
    x = torch.randn(M, K, device=DEV, generator=g).half()
    w = (0.02 * torch.randn(N, K, device=DEV, generator=g)).half()
    ref = x.float() @ w.float().T
    sb = gs.gs_linear_scratch_bytes(M, N, split)
    stream = torch.cuda.current_stream().cuda_stream
    for _ in range(2):                     # stale bytes, then the previous call's leftovers
        y = torch.full((M, N), 7.0, dtype=torch.float16, device=DEV)
        if _ == 0:
            scratch = torch.full((sb,), 0x7F, dtype=torch.uint8, device=DEV)
        gs.gs_linear(x.data_ptr(), w.data_ptr(), y.data_ptr(), M, N, K, gs.EPI_STORE_F16, split,
                     scratch.data_ptr(), sb, stream)
        torch.cuda.synchronize()
        torch.testing.assert_close(y.float(), ref, rtol=2e-3, atol=1e-3 * ref.abs().max().item())
        assert int(scratch[:4].view(torch.int32).item()) == 0


@pytest.mark.parametrize("M,split", [(9, 1), (17, 2), (200, 1)])
def test_linear_swiglu(gs, M, split):
    F, K = 1024, 256
    g = torch.Generator(device=DEV).manual_seed(3)
    x = torch.randn(M, K, device=DEV, generator=g).half()
    w = (0.05 * torch.randn(2 * F, K, device=DEV, generator=g)).half()
    gu = x.float() @ w.float().T
    ref = torch.nn.functional.silu(gu[:, :F]) * gu[:, F:]
    y = torch.zeros(M, F, dtype=torch.float16, device=DEV)
    _linear(gs, x, w, M, F, K, gs.EPI_SWIGLU, split, y)
    torch.testing.assert_close(y.float(), ref, rtol=2e-3, atol=1e-3 * ref.abs().max().item())


@pytest.mark.parametrize("M,V", [(1, 4096), (17, 59392), (70, 4096)])
def test_linear_argmax(gs, M, V):
    K = 1024
    g = torch.Generator(device=DEV).manual_seed(M)
    x = torch.randn(M, K, device=DEV, generator=g).half()
    w = (0.02 * torch.randn(V, K, device=DEV, generator=g)).half()
    ref = x.float() @ w.float().T
    keys = torch.zeros(M, dtype=torch.int64, device=DEV)
    _linear(gs, x, w, M, V, K, gs.EPI_ARGMAX, 1, keys)
    idx = (0xFFFFFFFF - (keys & 0xFFFFFFFF)).cpu().numpy()
    want = ref.argmax(dim=1).cpu().numpy()
    top2 = ref.topk(2, dim=1).values
    gap = (top2[:, 0] - top2[:, 1]).cpu().numpy()
    for i in range(M):
        if idx[i] != want[i]:
            assert gap[i] < 1e-4, (i, idx[i], want[i], gap[i])
    # ties resolve to the lowest index: duplicate the winning row further down
    w2 = w.clone()
    w2[V - 1] = w2[int(want[0])]
    keys.zero_()
    _linear(gs, x[:1].contiguous(), w2, 1, V, K, gs.EPI_ARGMAX, 1, keys)
    got = int(0xFFFFFFFF - (int(keys[0].item()) & 0xFFFFFFFF))
    assert got == min(int(want[0]), V - 1) or gap[0] < 1e-4


def test_linear_rows_do_not_depend_on_batch(gs):
    """Same token tile and split: a row's bits do not depend on the other rows."""
    N, K = 2048, 1024
    g = torch.Generator(device=DEV).manual_seed(5)
    x = torch.randn(17, K, device=DEV, generator=g).half()
    w = (0.02 * torch.randn(N, K, device=DEV, generator=g)).half()
    y17 = torch.zeros(17, N, dtype=torch.float16, device=DEV)
    _linear(gs, x, w, 17, N, K, gs.EPI_STORE_F16, 8, y17)
    for r in (0, 5, 16):
        y1 = torch.zeros(1, N, dtype=torch.float16, device=DEV)
        _linear(gs, x[r:r + 1].contiguous(), w, 1, N, K, gs.EPI_STORE_F16, 8, y1)
        assert torch.equal(y1[0], y17[r])


@pytest.mark.parametrize("split", [1, 2, 8])
def test_linear_rows_do_not_depend_on_tile_width(gs, split):
    """Same split-K factor, different token counts (token tiles of 32, 64, 128
    and 256 columns): the first rows' bits are the same."""
    N, K = 1024, 1024
    g = torch.Generator(device=DEV).manual_seed(11)
    x = torch.randn(300, K, device=DEV, generator=g).half()
    w = (0.02 * torch.randn(N, K, device=DEV, generator=g)).half()
    ys = {}
    for M in (17, 40, 100, 300):
        y = torch.zeros(M, N, dtype=torch.float16, device=DEV)
        _linear(gs, x[:M].contiguous(), w, M, N, K, gs.EPI_STORE_F16, split, y)
        ys[M] = y
        r = torch.zeros(M, N, dtype=torch.float32, device=DEV)
        _linear(gs, x[:M].contiguous(), w, M, N, K, gs.EPI_RESID_F32, split, r)
        ys[(M, "f32")] = r
    for M in (40, 100, 300):
        assert torch.equal(ys[M][:17], ys[17]), M
        assert torch.equal(ys[(M, "f32")][:17], ys[(17, "f32")]), M


# ------------------------------------------------------------------ attention
def _paged(k, v, rng):
    """Pack per-sequence K/V [B, ctx, Hkv, 64] into a shuffled page pool: per
    page and KV head, K as [token][dim] and V transposed as [dim][token]."""
    B, ctx, Hkv, hd = k.shape
    pages_per = math.ceil(ctx / 64)
    n_pages = B * pages_per + 3
    perm = rng.permutation(n_pages)[: B * pages_per].reshape(B, pages_per)
    pool = np.zeros((n_pages, 2, Hkv, 64, 64), dtype=np.float16)
    for b in range(B):
        for p in range(pages_per):
            t0, t1 = p * 64, min(ctx, p * 64 + 64)
            pool[perm[b, p], 0, :, : t1 - t0] = k[b, t0:t1].transpose(1, 0, 2)      # [head][tok][dim]
            pool[perm[b, p], 1, :, :, : t1 - t0] = v[b, t0:t1].transpose(1, 2, 0)   # [head][dim][tok]
    return pool, perm.astype(np.int32), n_pages


def _oracle_attn(q, k, v, allowed, Hq, Hkv):
    fake = types.SimpleNamespace(cfg=types.SimpleNamespace(n_heads=Hq, n_kv_heads=Hkv, head_dim=64))
    return Decoder.attention(fake, q, k, v, allowed)


def _run_attention(gs, mode, q, pool, pt, n_arr, W, Hq, Hkv, split_pages):
    B = q.shape[0]
    qd = torch.from_numpy(q).to(DEV)
    kvd = torch.from_numpy(pool).to(DEV)
    ptd = torch.from_numpy(pt).to(DEV)
    nd = torch.from_numpy(n_arr.astype(np.int32)).to(DEV)
    out = torch.zeros(q.shape, dtype=torch.float16, device=DEV)
    sb = gs.gs_attention_scratch_bytes(B, W, Hq, Hkv, pt.shape[1], split_pages)
    scratch = torch.zeros(sb, dtype=torch.uint8, device=DEV)
    gs.gs_attention(mode, qd.data_ptr(), kvd.data_ptr(), pool.shape[0], ptd.data_ptr(), pt.shape[1],
                    nd.data_ptr(), B, W, Hq, Hkv, out.data_ptr(), scratch.data_ptr(), sb,
                    split_pages, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return out.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("W,ns,Hq,Hkv,sp", [
    (5, [1, 63, 64], 16, 8, 1),
    (17, [2048, 2500], 16, 8, 2),
    (33, [0, 127, 4000], 16, 8, 3),
    (65, [190, 1030], 16, 8, 64),
    (9, [440, 511], 4, 4, 2),
])
def test_attention_matches_oracle(gs, mode, W, ns, Hq, Hkv, sp):
    rng = np.random.default_rng(W * 31 + mode)
    B = len(ns)
    ctx = max(ns) + W + 1
    q, k, v = synth.attn_inputs(B, W, ctx, Hq, Hkv, index=W + mode)
    pool, pt, n_pages = _paged(k, v, rng)
    got = _run_attention(gs, mode, q, pool, pt, np.array(ns), W, Hq, Hkv, sp)
    K = W - 1
    for b, n in enumerate(ns):
        allowed = od.draft_allowed(n, K) if mode == 0 else od.verify_allowed(n, K)
        nk = allowed.shape[1]
        want = _oracle_attn(q[b].astype(np.float64), k[b, :nk].astype(np.float64),
                            v[b, :nk].astype(np.float64), allowed, Hq, Hkv)
        np.testing.assert_allclose(got[b], want, rtol=5e-3, atol=5e-3)


@pytest.mark.parametrize("B,prefix,K", [(64, 8192, 64), (8, 4096, 16), (1, 1024, 4)])
def test_attention_sweep_sizes_sampled(gs, B, prefix, K):
    """Attention-sweep shapes; the oracle checks a seeded sample of sequences."""
    W = K + 1
    Hq, Hkv = 16, 8
    rng = np.random.default_rng(prefix + B)
    ns = [prefix] * B
    ctx = prefix + W + 1
    q, k, v = synth.attn_inputs(B, W, ctx, Hq, Hkv, index=B)
    pool, pt, _ = _paged(k, v, rng)
    sp = max(2, math.ceil(pt.shape[1] / 8))   # the engine's default: at most 8 items
    for mode in (0, 1):
        got = _run_attention(gs, mode, q, pool, pt, np.array(ns), W, Hq, Hkv, sp)
        for b in sorted(set([0, B - 1] + list(rng.integers(0, B, 2)))):
            allowed = od.draft_allowed(prefix, K) if mode == 0 else od.verify_allowed(prefix, K)
            nk = allowed.shape[1]
            want = _oracle_attn(q[b].astype(np.float64), k[b, :nk].astype(np.float64),
                                v[b, :nk].astype(np.float64), allowed, Hq, Hkv)
            np.testing.assert_allclose(got[b], want, rtol=5e-3, atol=5e-3)


@pytest.mark.parametrize("sp", [3, 1])
def test_attention_rows_do_not_depend_on_window(gs, sp):
    """Verify mode: the rows of a 17-token window and the first 17 rows of a
    33- and a 65-token window (two query blocks of 128 rows) over the same
    cache have the same limits and queries, so the same bits -- with the
    items merged in a cluster (sp = 3: at most 8 items) or through global
    scratch (sp = 1: 11 items)."""
    Hq, Hkv, n = 16, 8, 620
    rng = np.random.default_rng(3)
    q, k, v = synth.attn_inputs(1, 65, n + 67, Hq, Hkv, index=77)
    pool, pt, _ = _paged(k, v, rng)
    outs = {}
    for W in (17, 33, 65):
        outs[W] = _run_attention(gs, 1, np.ascontiguousarray(q[:, :W]), pool, pt, np.array([n]), W,
                                 Hq, Hkv, sp)
    assert np.array_equal(outs[33][:, :17], outs[17])
    assert np.array_equal(outs[65][:, :17], outs[17])
    assert np.array_equal(outs[65][:, :33], outs[33])

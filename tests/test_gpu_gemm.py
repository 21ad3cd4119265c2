"""The whole layer's projections on the tcgen05 GEMM (kvr_linear,
kvr_linear_swiglu) against the oracle's projection steps (fp64 product of the
same bf16 inputs, one rounding), at shapes with ragged row, column and K tails,
both tile widths (128 columns up to 512 rows, 256 above), the residual input,
and the Qwen3-4B layer's widths on sampled rows."""
import numpy as np
import pytest

import oracle
from harness import bits_of, tdev
from paper_2606_13361_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def kvr():
    from paper_2606_13361_gb300 import kvr as k
    assert torch.cuda.is_available()
    return k


@pytest.fixture(scope="module")
def ctx(kvr):
    C = kvr.Context(kvr.make_desc(1, 4, 1, 64, 1024), n_pages=2, max_seqs=2)
    yield C
    C.close()


def _ulp(v):
    """bf16 spacing at |v| (the smallest normal spacing below 2^-126)."""
    e = np.floor(np.log2(np.maximum(np.abs(v), 2.0 ** -126)))
    return 2.0 ** (e - 7)


def _check(got_bits, want_bits, exact, ulps, min_equal, what, acc=0.0):
    """got within `ulps` bf16 spacings of the fp64 value plus `acc` (a bound
    on the fp32 accumulation error), and at least min_equal of the elements
    equal to the oracle's own rounding."""
    got = oracle.bf16_decode(got_bits)
    err = np.abs(got - exact)
    bound = ulps * _ulp(exact) + acc
    assert np.all(err <= bound), f"{what}: worst {err.max():.3g} at {np.unravel_index(np.argmax(err - bound), err.shape)}"
    eq = float(np.mean(got_bits == want_bits))
    assert eq >= min_equal, f"{what}: {eq:.4f} of the elements equal the oracle's rounding"


@pytest.mark.parametrize("T,N,K,res,split", [
    (200, 520, 264, True, False),     # row, column and K tails; 128-wide tiles
    (9, 256, 128, False, False),      # just above the decode-size GEMV
    (1, 64, 64, True, False),         # one row
    (513, 1024, 2560, True, False),   # 256-wide tiles, one row past a tile
    (700, 6144, 2560, False, False),  # the fused q/k/v width
    (64, 2560, 4096, True, True),     # a q = 64 continuation's output projection: K split over CTAs
    (100, 520, 1000, False, True),    # split K with a K tail and a column tail
])
def test_linear_matches_oracle(kvr, ctx, T, N, K, res, split):
    x = inputs.normal_bf16(80 + T, (T, K))
    w = inputs.normal_bf16(81 + N, (N, K))
    c = inputs.normal_bf16(82, (T, N)) if res else None
    out = torch.empty((T, N), dtype=torch.bfloat16, device="cuda")
    ws = torch.full(((16 << 20) // 4,), float("nan"), dtype=torch.float32, device="cuda") if split else None
    n0 = kvr.kvr_launch_count(ctx.ctx)
    kvr.kvr_linear(ctx.ctx, tdev(x), tdev(w), out, tdev(c) if res else None, workspace=ws)
    assert kvr.kvr_launch_count(ctx.ctx) - n0 == (2 if split else 1)  # split: the GEMM and the reduction
    assert kvr.kvr_sync_status(ctx.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
    got = bits_of(out)
    rows = np.arange(T) if T <= 256 else np.random.default_rng(T).choice(T, 256, replace=False)
    xf, wf = oracle.bf16_decode(x[rows]), oracle.bf16_decode(w)
    exact = xf @ wf.T + (oracle.bf16_decode(c[rows]) if res else 0.0)
    want = oracle.linear(x[rows], w, c[rows] if res else None)
    # one rounding of an fp32 sum (half an ulp of that sum) plus the fp32
    # accumulation error, at most K 2^-24 sum |x w| (with the residual: one
    # more term)
    acc = (K + 1) * 2.0 ** -24 * (np.abs(xf) @ np.abs(wf).T + (np.abs(oracle.bf16_decode(c[rows])) if res else 0.0))
    _check(got[rows], want, exact, 0.5, 0.99, f"linear T={T} N={N} K={K}", acc=acc)


@pytest.mark.parametrize("T,I,K,split", [(200, 264, 136, False), (600, 9728, 2560, False), (40, 512, 2560, False),
                                         (40, 512, 2560, True), (64, 9728, 2560, True)])
def test_linear_swiglu_matches_oracle(kvr, ctx, T, I, K, split):
    x = inputs.normal_bf16(90 + T, (T, K))
    # weights at the scale of a trained projection (N(0, 1/K)) so silu is not saturated
    wgu = inputs.to_bf16_bits((np.random.default_rng(91).standard_normal((2 * I, K)) / np.sqrt(K)).astype(np.float32))
    out = torch.empty((T, I), dtype=torch.bfloat16, device="cuda")
    ws = torch.full(((16 << 20) // 4,), float("nan"), dtype=torch.float32, device="cuda") if split else None
    kvr.kvr_linear_swiglu(ctx.ctx, tdev(x), tdev(wgu), out, workspace=ws)
    assert kvr.kvr_sync_status(ctx.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
    got = bits_of(out)
    rows = np.arange(T) if T <= 256 else np.random.default_rng(T).choice(T, 256, replace=False)
    want = oracle.linear_swiglu(x[rows], wgu[:I], wgu[I:])
    assert float(np.mean(got[rows] == want)) >= 0.98
    # g and u are bf16 roundings of sums that the GPU forms in fp32: each lies
    # within K 2^-24 sum |x w| (the fp32 accumulation bound) plus one bf16 step
    # of the exact sum (near cancellation the first term dominates).  Every
    # GPU value lies within one bf16 step of the range that silu(g) u takes
    # over those intervals.
    xf = oracle.bf16_decode(x[rows])
    ivals = []
    for wpart in (wgu[:I], wgu[I:]):
        wf = oracle.bf16_decode(wpart)
        ex = xf @ wf.T
        rad = K * 2.0 ** -24 * (np.abs(xf) @ np.abs(wf).T) + _ulp(ex)
        ivals.append((ex - rad, ex + rad))
    (gl, gh), (ul, uh) = ivals
    s_min = np.minimum(oracle.silu(gl), oracle.silu(gh))
    s_max = np.maximum(oracle.silu(gl), oracle.silu(gh))
    gmin = -1.2784645427610738  # silu's minimum (1 + g + e^g = 0): inside the interval it is the lowest value
    inside = (gl < gmin) & (gh > gmin)
    s_min = np.where(inside, oracle.silu(np.array(gmin)), s_min)
    prods = [s_min * ul, s_min * uh, s_max * ul, s_max * uh]
    lo, hi = np.min(prods, axis=0), np.max(prods, axis=0)
    a = oracle.bf16_decode(got[rows])
    tol = _ulp(np.maximum(np.abs(lo), np.abs(hi)))
    bad = (a < lo - tol) | (a > hi + tol)
    if bad.any():
        r_, c_ = np.nonzero(bad)
        ex = [(int(rows[i]), int(j), float(a[i, j]), float(lo[i, j]), float(hi[i, j])) for i, j in zip(r_[:12], c_[:12])]
        raise AssertionError(f"swiglu T={T} I={I} K={K}: {int(bad.sum())} values outside the bound; "
                             f"(row, col, gpu, lo, hi): {ex}")


def test_linear_rejects_bad_shapes(kvr, ctx):
    x = torch.zeros((16, 60), dtype=torch.bfloat16, device="cuda")
    w = torch.zeros((64, 60), dtype=torch.bfloat16, device="cuda")
    out = torch.empty((16, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvr.KvrError) as e:  # K not a multiple of 8
        kvr.kvr_linear(ctx.ctx, x, w, out)
    assert e.value.status == kvr.KVR_ERR_INVALID_ARG
    buf = torch.zeros(16 * 64 + 1, dtype=torch.bfloat16, device="cuda")
    x2 = buf[1:].view(16, 64)  # 2-byte offset: not 16-byte aligned
    w2 = torch.zeros((64, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvr.KvrError) as e:
        kvr.kvr_linear(ctx.ctx, x2, w2, out)
    assert e.value.status == kvr.KVR_ERR_INVALID_ARG
    assert kvr.kvr_sync_status(ctx.ctx) == kvr.KVR_OK

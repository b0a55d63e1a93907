"""The two-part bf16 split behind the fp32 path's tensor-core contractions, on CPU.

An fp32 value x is split as hi = bf16(x) (round to nearest even) and lo = bf16(x - hi);
a contraction sum_k a_k b_k is then formed from three bf16 products per term,
a_hi b_hi + a_hi b_lo + a_lo b_hi, each exact in fp32, accumulated in fp32.  The fp32
path's gate and head GEMMs (three passes into one TMEM accumulator) and the training
step's recurrence GEMM (one bf16 GEMM over K = 3 * 4H) both rely on it.

bf16 keeps 8 significant bits, so its unit roundoff is u = 2^-8: |x - hi| <= u |x|,
x - hi is exact in fp32, and the part lo leaves a residual of at most u |x - hi| <= u^2 |x|.
The dropped terms per product (a_lo b_lo and the two residuals against the other
operand's hi part, plus smaller ones) therefore total at most about 3 u^2 |a b|,
whatever the values: the bound checked here, with the sums themselves taken in fp64.
"""
import numpy as np
import pytest
import torch

U = 2.0 ** -8
BOUND = 3.0 * U * U * (1.0 + 4.0 * U)  # 3 u^2 and the higher-order terms


def _bf16(x32: np.ndarray) -> np.ndarray:
    """bf16 round-to-nearest-even of fp32 values, returned as fp32."""
    return torch.from_numpy(np.ascontiguousarray(x32, dtype=np.float32)).to(torch.bfloat16).float().numpy()


def _split(x32: np.ndarray):
    hi = _bf16(x32)
    d = (x32 - hi).astype(np.float32)  # exact in fp32
    return hi, _bf16(d), d


def _draw(kind: str, n: int, rng) -> np.ndarray:
    if kind == "normal":
        x = rng.standard_normal(n)
    elif kind == "uniform":
        x = rng.uniform(-1.0, 1.0, n)
    elif kind == "wide":  # magnitudes over 2^-20 .. 2^20, both signs
        x = rng.choice([-1.0, 1.0], n) * np.exp2(rng.uniform(-20.0, 20.0, n))
    else:  # gradients of a cell: small values, many near zero
        x = 1e-3 * rng.standard_normal(n) * (rng.random(n) < 0.7)
    return x.astype(np.float32)


def test_split_parts_are_exact_and_small():
    rng = np.random.default_rng(7)
    for kind in ("normal", "uniform", "wide", "grad"):
        x = _draw(kind, 4096, rng)
        hi, lo, d = _split(x)
        # x - hi is representable in fp32: the fp32 difference equals the exact one
        np.testing.assert_array_equal(d.astype(np.float64), x.astype(np.float64) - hi.astype(np.float64))
        ax = np.abs(x.astype(np.float64))
        assert np.all(np.abs(d.astype(np.float64)) <= U * ax)
        resid = d.astype(np.float64) - lo.astype(np.float64)
        assert np.all(np.abs(resid) <= U * U * ax)


@pytest.mark.parametrize("K", [16, 576, 2048, 6144])
@pytest.mark.parametrize("kinds", [("normal", "normal"), ("uniform", "grad"), ("wide", "normal"),
                                   ("grad", "wide")])
def test_three_products_stay_within_the_bound(K, kinds):
    rng = np.random.default_rng(K)
    for _ in range(8):
        a, b = _draw(kinds[0], K, rng), _draw(kinds[1], K, rng)
        ah, al, _ = _split(a)
        bh, bl, _ = _split(b)
        a64, b64 = a.astype(np.float64), b.astype(np.float64)
        exact = np.dot(a64, b64)
        three = (np.dot(ah.astype(np.float64), bh.astype(np.float64)) +
                 np.dot(ah.astype(np.float64), bl.astype(np.float64)) +
                 np.dot(al.astype(np.float64), bh.astype(np.float64)))
        scale = np.dot(np.abs(a64), np.abs(b64))
        assert abs(three - exact) <= BOUND * scale


def test_dropping_a_cross_term_breaks_the_bound():
    # hi.hi + hi.lo alone (a mistake: the lo.hi pass left out).  With a_k = 1 + 2^-10 every
    # lo part is +2^-10 (below half a bf16 ulp of 1), so the missing term is 2^-10 sum b_k,
    # about 20 times the bound
    rng = np.random.default_rng(3)
    a = np.full(2048, 1.0 + 2.0 ** -10, dtype=np.float32)
    b = rng.uniform(0.5, 1.0, 2048).astype(np.float32)
    ah, al, _ = _split(a)
    bh, bl, _ = _split(b)
    assert np.all(al == np.float32(2.0 ** -10))
    a64, b64 = a.astype(np.float64), b.astype(np.float64)
    exact = np.dot(a64, b64)
    two = np.dot(ah.astype(np.float64), bh.astype(np.float64)) + np.dot(ah.astype(np.float64), bl.astype(np.float64))
    three = two + np.dot(al.astype(np.float64), bh.astype(np.float64))
    scale = np.dot(np.abs(a64), np.abs(b64))
    assert abs(two - exact) > 10 * BOUND * scale
    assert abs(three - exact) <= BOUND * scale


def test_concatenated_operands_give_the_three_products():
    # the recurrence GEMM's layout: A rows [hi | hi | lo], B rows [hi | lo | hi] over K = 3 * n
    rng = np.random.default_rng(11)
    g, w = _draw("grad", 512, rng), _draw("normal", 512, rng)
    gh, gl, _ = _split(g)
    wh, wl, _ = _split(w)
    arow = np.concatenate([gh, gh, gl]).astype(np.float64)
    brow = np.concatenate([wh, wl, wh]).astype(np.float64)
    three = (np.dot(gh.astype(np.float64), wh.astype(np.float64)) + np.dot(gh.astype(np.float64), wl.astype(np.float64)) +
             np.dot(gl.astype(np.float64), wh.astype(np.float64)))
    assert np.dot(arow, brow) == pytest.approx(three, rel=1e-15, abs=1e-300)

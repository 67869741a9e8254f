"""The parity bar itself (tests/parity.py), on the CPU: each planted mistake
in a 'GPU' result fails it, and values exactly at the bar pass."""
import numpy as np
import pytest
import torch

from tests.parity import BF16_CAST, check_values


def _base():
    want = np.array([1.0, -2.0, 0.5, 0.0, 3.0])
    mag = np.array([2.0, 4.0, 1.0, 0.0, 3.0])
    return want.copy(), want, mag


def test_exact_result_passes():
    g, want, mag = _base()
    assert check_values(g, want, mag, torch.float32, False) == 0.0


def test_planted_nan_fails():
    g, want, mag = _base()
    g[1] = np.nan
    with pytest.raises(AssertionError, match="finite"):
        check_values(g, want, mag, torch.bfloat16, True)


def test_planted_inf_fails():
    g, want, mag = _base()
    g[2] = np.inf
    with pytest.raises(AssertionError, match="finite"):
        check_values(g, want, mag, torch.float32, False)


def test_wrong_sign_inf_fails():
    want = np.array([np.inf, -np.inf, np.nan, 1.0])
    mag = np.array([np.inf, np.inf, np.nan, 1.0])
    check_values(want.copy(), want, mag, torch.float32, False)
    g = want.copy()
    g[0] = -np.inf
    with pytest.raises(AssertionError, match="non-finite"):
        check_values(g, want, mag, torch.float32, False)
    g = want.copy()
    g[2] = np.inf
    with pytest.raises(AssertionError, match="non-finite"):
        check_values(g, want, mag, torch.float32, False)


def test_error_just_above_bound_fails():
    g, want, mag = _base()
    tol = 1e-5
    g[0] = want[0] + tol * mag[0] * (1 - 1e-9)
    check_values(g, want, mag, torch.float32, False)
    g[0] = want[0] + tol * mag[0] * (1 + 1e-6)
    with pytest.raises(AssertionError, match="out of tolerance"):
        check_values(g, want, mag, torch.float32, False)


def test_nonzero_where_no_contribution_fails():
    g, want, mag = _base()
    g[3] = 1e-30
    with pytest.raises(AssertionError, match="exactly zero"):
        check_values(g, want, mag, torch.float32, False)


def test_scale_widens_the_bound():
    g, want, mag = _base()
    g[4] = want[4] + 1.5e-5 * mag[4]
    with pytest.raises(AssertionError):
        check_values(g, want, mag, torch.float32, False)
    check_values(g, want, mag, torch.float32, False, scale=2.0)


def test_bf16_cast_term_is_the_unit_roundoff():
    """1 + 2^-8 is a tie between bf16 neighbours 1 and 1 + 2^-7 and rounds to
    1: a correct cast errs by 2^-8 / (1 + 2^-8) of the value, which a 2^-9
    term would reject."""
    x = 1.0 + 2.0**-8
    cast = torch.tensor([x], dtype=torch.float32).to(torch.bfloat16).double().item()
    assert cast == 1.0
    want = np.array([x])
    mag = np.array([1e-12])          # accumulation bound ~0: the cast term alone
    check_values(np.array([cast]), want, mag, torch.float32, True)
    assert abs(cast - x) > 2.0**-9 * x
    assert abs(cast - x) <= BF16_CAST * x
    with pytest.raises(AssertionError):
        check_values(np.array([cast - 2.0**-14]), want, mag, torch.float32, True)
    with pytest.raises(AssertionError):   # no cast term for an fp32 output
        check_values(np.array([cast]), want, mag, torch.float32, False)


def test_bf16_reaches_oracle_workers_exactly():
    """bf16 tiles travel to the oracle workers as raw 16-bit patterns and are
    widened there: every pattern (signed zeros, infinities, NaN, subnormals)
    must come out equal to torch's own bf16 -> float32 conversion."""
    from tests.parity import _to_worker, _widen
    bits = torch.arange(-32768, 32768, dtype=torch.int32).to(torch.int16)
    t = bits.view(torch.bfloat16)
    got = _widen(_to_worker(t))
    want = t.float().numpy()
    assert got.dtype == np.float32
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


def test_oracle_parallel_matches_oracle_ref():
    """The spawned-pool path gives the same oracle result as a direct call,
    for bf16 and fp32 tiles, with sampled keys."""
    from tests.parity import oracle_parallel, oracle_ref
    g = torch.Generator().manual_seed(2)
    ka = np.array([[0, 0], [0, 1], [1, 1], [2, 0]], np.int32)
    kb = np.array([[0, 0], [1, 0], [1, 2]], np.int32)
    ta = torch.randn((4, 4, 3), generator=g).to(torch.bfloat16)
    tb = torch.randn((3, 3, 5), generator=g)
    rels = [(ka, (3, 2), ta), (kb, (2, 3), tb)]
    spec = "IiJj,JjKk->IiKk"
    direct = oracle_ref(spec, rels, sample_keys=np.array([[0, 0], [2, 2]], np.int32))
    (pooled,) = oracle_parallel([(spec, rels, {"sample_keys": np.array([[0, 0], [2, 2]], np.int32)})])
    assert np.array_equal(direct["keys"], pooled["keys"])
    assert np.array_equal(direct["out"], pooled["out"]) and np.array_equal(direct["abs"], pooled["abs"])

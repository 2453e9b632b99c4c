"""Dispatch-ratio feedback (Sec. 3.4): the host controller that picks the
decode share of the next step from the phase times of the last one. Host
arithmetic only; no GPU."""
import pytest

import paper_2606_04415_gb300 as fnpu


def test_share_kept_inside_tolerance():
    assert fnpu.dispatch_next_share(24, 1.00, 0.97, tolerance=0.05) == 24
    assert fnpu.dispatch_next_share(24, 1.00, 1.04, tolerance=0.05) == 24


def test_share_moves_toward_the_side_that_ends_later():
    # decode ends much later: more SMs to decode; much earlier: fewer
    assert fnpu.dispatch_next_share(20, 1.0, 2.0, tolerance=0.05) > 20
    assert fnpu.dispatch_next_share(20, 2.0, 1.0, tolerance=0.05) < 20
    # outside the band it always moves at least one point
    assert fnpu.dispatch_next_share(20, 1.0, 1.07, tolerance=0.05) == 21


@pytest.mark.parametrize("d_work,p_work", [(0.3, 1.5), (1.0, 1.0), (0.05, 2.0), (0.8, 0.4)])
def test_share_converges_on_a_split_sm_model(d_work, p_work):
    """Times of a device where each phase holds its own SMs: decode d/s,
    prefill p/(1 - s). The loop settles where both end together, s* =
    d/(d + p), within the tolerance band (clamped to [1, 50] %)."""
    s = 24
    for _ in range(40):
        dec, pre = d_work / (s / 100), p_work / (1 - s / 100)
        s = fnpu.dispatch_next_share(s, pre, dec, tolerance=0.03)
    target = min(max(100 * d_work / (d_work + p_work), 1), 50)
    dec, pre = d_work / (s / 100), p_work / (1 - s / 100)
    assert abs(dec - pre) <= 0.03 * max(dec, pre) or abs(s - target) <= 1 or s in (1, 50)
    assert abs(s - target) <= 2.5
    # settled: one more step keeps it
    assert fnpu.dispatch_next_share(s, pre, dec, tolerance=0.03) == s


def test_share_is_clamped():
    assert fnpu.dispatch_next_share(50, 0.1, 100.0, tolerance=0.0) == 50
    assert fnpu.dispatch_next_share(1, 100.0, 0.1, tolerance=0.0) == 1
    assert fnpu.dispatch_next_share(80, 1.0, 1.0, tolerance=0.1) == 50  # kept, but within range


@pytest.mark.parametrize("args", [(0, 1.0, 1.0, 0.05), (100, 1.0, 1.0, 0.05), (20, 0.0, 1.0, 0.05),
                                  (20, 1.0, -1.0, 0.05), (20, 1.0, 1.0, -0.1), (20, float("nan"), 1.0, 0.05)])
def test_controller_rejects_bad_arguments(args):
    with pytest.raises(fnpu.FnpuError) as e:
        fnpu.dispatch_next_share(*args)
    assert e.value.code == fnpu.FNPU_EINVAL


def test_phase_times_reject_a_null_plan():
    import ctypes
    a, b = ctypes.c_float(), ctypes.c_float()
    assert fnpu.load().fnpu_plan_phase_ms(None, ctypes.byref(a), ctypes.byref(b)) == fnpu.FNPU_EINVAL

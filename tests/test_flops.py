"""Pins of the App. G prefill-FLOPs accounting (Eqs. perlayer, prefill, ratio)."""

import pytest

from paper_2608_08794_gb300 import flops as F


def test_phi_closed_form_for_the_7b_thinker():
    # phi(1000) = 4*1000*3584^2 + 2*1000^2*3584 + 2*1000*3584*18944, worked by hand:
    #   4*1000*12845056      =  51 380 224 000
    #   2*1000000*3584       =   7 168 000 000
    #   2*1000*3584*18944    = 135 790 592 000
    assert F.phi(1000, F.QWEN25_OMNI_7B) == 51_380_224_000 + 7_168_000_000 + 135_790_592_000
    assert F.phi(0, F.QWEN25_OMNI_7B) == 0.0
    # the attention term is the only quadratic one
    m = F.QWEN25_OMNI_3B
    lin = F.phi(1, m) - 2 * m.hidden
    assert F.phi(10, m) == pytest.approx(10 * lin + 2 * 100 * m.hidden)


def test_constant_schedule_has_ratio_one_and_full_cost():
    m = F.QWEN25_OMNI_7B
    sched = F.layer_schedule(9000, [], m)
    assert sched == [9000] * 28
    assert F.flops_ratio(sched, 9000, m) == pytest.approx(1.0)
    assert F.prefill_flops(sched, m) == pytest.approx(28 * F.phi(9000, m))


def test_pruning_layer_runs_at_its_entering_length():
    m = F.QWEN25_OMNI_7B
    sched = F.layer_schedule(100, [(4, 50), (12, 20)], m)
    assert sched[:5] == [100] * 5 and sched[5:13] == [50] * 8 and sched[13:] == [20] * 15
    expect = (5 * F.phi(100, m) + 8 * F.phi(50, m) + 15 * F.phi(20, m)) / (28 * F.phi(100, m))
    assert F.flops_ratio(sched, 100, m) == pytest.approx(expect)
    with pytest.raises(ValueError):
        F.prefill_flops([1, 2, 3], m)


def test_paper_reduction_figure_is_a_ratio_of_its_table_values():
    # Table main7b: 67.9 T at full tokens, 15.0 T for the 25% tier ("up to 78%").
    assert 1 - 15.0 / 67.9 == pytest.approx(0.779, abs=1e-3)

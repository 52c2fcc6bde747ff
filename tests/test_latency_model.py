"""Rule-based block-size selection (Sec. 5.2): the rule on given latency
tables (CPU), and one small measured setting (GPU)."""
import pytest

from paper_2111_11581_gb300 import latency_model as lm


def _table(setting, lat):
    return {setting.key(): dict(lat)}


def test_scheme_mapping_follows_the_decision_tree():
    assert lm.scheme_for("dw3x3") is None
    assert lm.scheme_for("conv3x3") == "punched"
    assert lm.scheme_for("conv1x1") == "based"
    assert lm.scheme_for("fc") == "based"
    assert lm.select_block({}, lm.Setting("dw3x3", 64, 64, 56, 8.0)) is None


def test_smallest_block_within_beta_is_chosen():
    s = lm.Setting("conv3x3", 64, 64, 56, 8.0)
    t = _table(s, {"structured": 1.0, "4x4": 1.50, "8x4": 1.21, "8x8": 1.19, "16x8": 1.05,
                   "32x32": 1.0})
    # 8x4 is 21 % slower (out), 8x8 19 % (in): the smallest valid block wins
    assert lm.select_block(t, s, beta=0.2) == (8, 8)
    # a looser threshold admits 8x4, a tighter one only 16x8 and 32x32
    assert lm.select_block(t, s, beta=0.25) == (8, 4)
    assert lm.select_block(t, s, beta=0.1) == (16, 8)
    # exactly at the threshold counts as within it
    assert lm.select_block(t, s, beta=0.5) == (4, 4)


def test_structured_when_no_block_is_fast_enough():
    s = lm.Setting("fc", 1000, 2048, 64, 6.0)
    t = _table(s, {"structured": 1.0, "8x8": 3.0, "32x32": 1.5})
    assert lm.select_block(t, s, beta=0.2) == lm.STRUCTURED


def test_ties_in_area_prefer_fewer_rows():
    s = lm.Setting("conv1x1", 256, 64, 56, 8.0)
    t = _table(s, {"structured": 1.0, "16x8": 1.1, "8x16": 1.1})
    assert lm.select_block(t, s) == (8, 16)


def test_candidates_fit_the_weight():
    c = lm.candidates("conv3x3", 16, 8)
    assert all(bm <= 16 and bk <= 8 for bm, bk in c if (bm, bk) != lm.STRUCTURED)
    assert c[-1] == lm.STRUCTURED and (8, 8) in c and (16, 16) not in c
    # block-based blocks may span the 1x1 layer's channels
    assert (128, 64) in lm.candidates("conv1x1", 256, 64)


@pytest.mark.gpu
def test_measured_setting_gives_every_candidate():
    s = lm.Setting("conv3x3", 32, 16, 14, 4.0, batch=8)
    row = lm.measure_setting(s, reps=3)
    names = {lm.block_name(b) for b in lm.candidates("conv3x3", 32, 16)}
    assert set(row) == names
    assert all(v > 0 for v in row.values())
    b = lm.select_block({s.key(): row}, s)
    assert b in lm.candidates("conv3x3", 32, 16)

"""The process-wide launch tuning (mk_attn_set_tuning / mk_attn_get_tuning):
range checks, defaults, and restoring on exit -- host only, no GPU."""
import pytest

from paper_2609_04523_gb300 import binding
from paper_2609_04523_gb300.build import build_library


@pytest.fixture(autouse=True)
def restore():
    build_library()
    yield
    binding.set_tuning()


def test_defaults():
    binding.set_tuning()
    assert binding.mk_attn_get_tuning().as_dict() == binding.DEFAULT_TUNING


@pytest.mark.parametrize("field, bad", [
    ("ctas", -1), ("ctas", 65536), ("schedule", -1), ("schedule", 4),
    ("rescale_log2", -0.5), ("rescale_log2", 16.5), ("rescale_log2", float("nan")),
    ("split_ctas_per_sm", 0), ("split_ctas_per_sm", 65), ("split_min_pages", 0),
    ("split_min_pages", 4097), ("mla_split_ctas_per_sm", 0), ("mla_split_ctas_per_sm", 65)])
def test_out_of_range_is_rejected_and_changes_nothing(field, bad):
    binding.set_tuning(ctas=77)
    t = binding.MkAttnTuning(**{**binding.DEFAULT_TUNING, field: bad})
    assert binding.mk_attn_set_tuning(t) == binding.MK_ERR_INVALID_ARG
    assert binding.mk_attn_get_tuning().ctas == 77


def test_null_restores_defaults_and_context_manager_restores_previous():
    binding.set_tuning(ctas=10, schedule=binding.SCHED_BLOCKED)
    with binding.tuning(rescale_log2=2.0, split_min_pages=16):
        t = binding.mk_attn_get_tuning()
        assert t.rescale_log2 == 2.0 and t.split_min_pages == 16 and t.ctas == 0
    t = binding.mk_attn_get_tuning()
    assert t.ctas == 10 and t.schedule == binding.SCHED_BLOCKED
    assert binding.mk_attn_set_tuning(None) == binding.MK_OK
    assert binding.mk_attn_get_tuning().as_dict() == binding.DEFAULT_TUNING


def test_unknown_field_is_an_error():
    with pytest.raises(ValueError):
        binding.set_tuning(tile_m=64)


def test_sweep_candidates_cover_the_space():
    from paper_2609_04523_gb300 import autotune
    space = {"ctas": [0, 76], "schedule": [0, 1, 2]}
    got = list(autotune.candidates(space))
    assert len(got) == 6 and {"ctas": 76, "schedule": 2} in got

"""The tensor-core rate probe (pf16_tc_rate) runs on the GPU and reports a
plausible kind::f16 rate: positive, and not far above the 16-bit dense
nominal (a rate far above it would mean the MMAs did not run)."""
import pytest

from paper_1911_07384_gb300 import pf16

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("n", [64, 256])
@pytest.mark.parametrize("f32", [False, True], ids=["f16acc", "f32acc"])
def test_tc_rate_probe(n, f32):
    tf = pf16.tc_rate(n, f32_accum=f32, chains=1, reps=4000)
    assert 10.0 < tf < 3000.0, tf
    assert pf16.sync_status() == 0

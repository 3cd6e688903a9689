"""The NVTX instrumentation hook of the training step, on the host: it names
each library call by kind and layer shape, passes arguments and results
through, and closes its range when the call raises."""
import pytest

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300.resnet50 import layer_label, nvtx_hook


class _Layer:
    def __init__(self, desc):
        self.desc = desc


def test_labels():
    assert layer_label(None) == "-"
    assert layer_label(_Layer(pf16.conv_desc(256, 56, 56, 64, 256, 1, 1, 1, 0))) == "256,56,56,64,256,1,1,1,0"
    assert layer_label(_Layer(pf16.bn_desc(256, 14, 14, 1024))) == "256,14,14,1024"


def test_hook_passes_through_and_closes_on_error():
    assert nvtx_hook("conv_fwd", None, lambda a, b=0: a + b, 2, b=3) == 5

    def boom():
        raise ValueError("x")

    with pytest.raises(ValueError):
        nvtx_hook("bn_fwd", None, boom)
    assert nvtx_hook("sgd", None, lambda: 7) == 7

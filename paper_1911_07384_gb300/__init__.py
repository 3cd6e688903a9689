"""pf16: pure-FP16 ResNet-50 training kernels for GB300 (sm_103a)."""

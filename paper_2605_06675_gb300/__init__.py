"""GB300-native (sm_103a) hot path of RateQuant (arXiv 2605.06675).

Per-head mixed-bit KV-cache quantization with bit-widths from reverse
waterfilling, variable-width bit-packing, a distortion-calibration sweep, and
split-K GQA decode attention that reads the packed cache directly.

The compute lives in ``librq.so`` (C ABI, ``include/rq.h``); ``rq`` is its
thin ctypes binding, ``path`` composes the calls, ``workloads`` and ``synth``
describe and draw the synthetic inputs.
"""
from . import rq  # noqa: F401

__all__ = ["rq"]

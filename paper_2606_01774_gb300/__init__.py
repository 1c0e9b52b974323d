"""FLARE block-denoising attention step on GB300 (sm_103a).

``flare`` is the ctypes binding of the C-ABI library ``libflare.so`` (built by
``build.build()``); ``workloads`` draws the seeded synthetic serving batches.
"""
from . import flare, workloads  # noqa: F401

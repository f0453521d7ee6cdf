"""Seeded synthetic inputs for the OccamToken prune path.

This package only draws random tensors with the shapes and value structure of
the paper's workloads (LLaVA-v1.5, LLaVA-NeXT, Qwen3-VL, video). It holds none
of the method's arithmetic: no softmax, no scores, no thresholds, no
compaction. Both the CPU oracle (through the tests) and the CUDA path (through
the tests and the bench) take their inputs from here.
"""

from .configs import CONFIGS, WORKLOADS, get_config  # noqa: F401
from .gen import make_batch, tiny_batch, batch_slice_to_host  # noqa: F401

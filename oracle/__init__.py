"""Float64 CPU oracle of the BCMT token mixer.

Test infrastructure only: the tests, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` use it to check and time the CUDA library.  The
library itself never imports it and has no CPU fallback.
"""

from .bcmt_oracle import backward, block_ranges, forward, forward_from_inputs  # noqa: F401

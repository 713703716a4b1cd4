"""GB300-native mixed prefill/decode paged attention (the iteration observed
by the Decode-Latency Feedback Prefill controller, arxiv 2609.38386).

The compute runs in ``libmixattn.so`` (hand-written CUDA for sm_103a, C ABI in
``include/mixattn.h``); this package is its ctypes binding plus the host-side
DLFP controller.  Creating a Context (or calling ``load()``) without the built
library raises ImportError: there is no fallback path.
"""
from ._binding import (EXPORTS, LIB_PATH, MX_OPT_DECODE_CTAS, MX_OPT_GRID, MX_OPT_PDL,  # noqa: F401
                       MX_OPT_PREFILL_PIECE_TILES, MX_OPT_SPLIT_KEYS, MX_OPT_TEST_STALL_BLOCK,
                       MX_OPT_V_STAGES, MX_OPT_WAIT_LIMIT_US, Context, MxError, load, plan_work)

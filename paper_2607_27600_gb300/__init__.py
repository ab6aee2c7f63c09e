"""Counter-causal KV-cache refresh (arXiv 2607.27600) on GB300 (sm_103a).

The CUDA library (libcc.so, C ABI in include/cc.h) scores every cached token
by counter-causal surprise (full pass or fast single-layer approximation),
selects the keep-set and compacts the cache in place.  `cc` is its Python
binding (one function per C entry point); `shard` splits one refresh over the
ranks of a torch.distributed group by query rows.
"""
from . import cc  # noqa: F401
from .cc import (CCError, Cache, Weights, SCORE_LOGIT, SCORE_LOGPROB, model_cfg,  # noqa: F401
                 load_library)

"""CPU oracle for the WaveZip condensation pass (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
and reference legs may import this package.  The product path never does.
"""
from .wavezip_oracle import *  # noqa: F401,F403
from .wavezip_oracle import (  # noqa: F401
    adaptive_avg_pool2d, allocate_budget, bilinear_resize, condense, cosine,
    daubechies_lowpass, decision_margins, dwt1d, dwt2d, dwt_len, extend_index,
    frame_filter, frame_relevance, global_budget, grid_shape, idwt1d, idwt2d,
    psi, query_embedding, saliency_map, token_saliency, visual_change,
    wavelet_filters, wsm, wta,
)

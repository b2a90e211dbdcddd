"""GB300 (sm_103a) implementation of the Similarity Chunk Rolling prefill hot path.

``scale`` binds the C ABI of ``libscale.so`` (declared in ``include/scale.h``);
``_build.build()`` compiles it in-tree with nvcc.
"""

from . import fidelity, scale  # noqa: F401
from ._build import build  # noqa: F401
from .scale import (  # noqa: F401
    SCALE_MODE_PER_CLUSTER,
    SCALE_MODE_PER_SUBCHUNK,
    ScaleError,
    ScaleLibraryMissing,
    ScaleParams,
    allocate,
    params,
    params_for,
    run_path,
)

"""Float64 CPU oracle for the dropless routed MoE layer.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this package.  The
product path (the CUDA library and its Python binding) never imports, links
or executes anything here, and this package imports nothing from the product.
"""
from .moe import *  # noqa: F401,F403
from .eq1 import *  # noqa: F401,F403
from .router_sigmoid import *  # noqa: F401,F403
from .shared import *  # noqa: F401,F403
from .fp8 import *  # noqa: F401,F403
from .nvfp4 import *  # noqa: F401,F403

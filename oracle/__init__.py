"""Plain CPU oracle for the Fairy2i widely-linear {+-1, +-i} layer.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline /
``--impl reference`` legs of ``bench.py`` may import this package. The product path (the CUDA
library and its Python binding) never imports, calls or links anything here, and this package
imports nothing from the product.

Everything is numpy, float64 unless a step is defined in float32 (see ``fairy2i_oracle``).
"""
from .fairy2i_oracle import *  # noqa: F401,F403

"""CPU oracle for the ACID hot path — TEST INFRASTRUCTURE ONLY.

Only the test suite, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU
baseline leg may import this package.  The product path (the CUDA library and
its Python binding) never imports, calls or links anything here.

Everything is plain numpy in float64.  Citations name the paper's sections,
equations and algorithm; where the paper is silent the docstring says which
reading is taken.

Parity-unpinned parts: the composition of the DiT blocks, the 3D RoPE axis
split and the EasyCache norms are readings (the paper names the models and
methods but defines none of them); their pins check internal consistency,
closed forms and library equivalence, not a statement of the paper.
"""

from .acid_oracle import *  # noqa: F401,F403

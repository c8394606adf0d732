"""GB300 (sm_103a) hot path of ACID, adaptive dual-threshold step caching
for video diffusion transformers: DiT block kernels, drift reductions and
the threshold-switching step loop behind a C ABI (include/acid.h).

``paper_2607_12358_gb300.acid`` is the Python binding; the library itself is
built by ``paper_2607_12358_gb300.build``.
"""

__all__ = ["acid", "build"]

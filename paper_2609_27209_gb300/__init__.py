"""ERC-LG on GB300: effective-resistance curvature of every edge of a large graph.

The computation runs in hand-written CUDA kernels behind the C ABI declared in ``include/erc.h``
(library ``liberc.so`` in this package).  ``paper_2609_27209_gb300.erc`` is the thin Python binding
with the same call names; it raises if the compiled library is missing -- there is no CPU path.
``paper_2609_27209_gb300.synth`` draws the seeded synthetic input graphs.
"""

"""CPU oracle for ERC-LG -- test infrastructure only.

Plain fp64 restatements of the paper's steps (``erc_oracle``) and dense small-graph definitions
(``dense``).  Only tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg may use
this package.  It shares no code with the CUDA library and never imports it.
"""

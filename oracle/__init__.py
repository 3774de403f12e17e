"""CPU oracle of AWSRC (arXiv 2608.23144) — TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s cpu_baseline leg
may import or run anything under ``oracle/``. The product path
(``paper_2608_23144_gb300``) never does, and the oracle never imports the
product package: the two share no code. The C source ``awsrc_oracle.c`` is the
oracle proper; ``oracle.py`` is argument marshalling around it.
"""

"""CPU oracle for the PSC vocabulary mask: test infrastructure, not part of the product.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import it.  It shares no code with the CUDA path.
"""
from .psc_oracle import Config, Oracle, OracleLimitError, Vocab, ST_OK, ST_DONE, ST_ERROR  # noqa: F401

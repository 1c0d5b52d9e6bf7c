"""GB300-native implementation of the hashed shared-array embedding (PSS with
ROBE-Z mapping) of "The trade-offs of model size in large recommendation
models" (Desai & Shrivastava, arXiv 2207.10731).

The compute path is the C-ABI library ``libpss.so`` built from ``csrc/``;
``paper_2207_10731_gb300.binding`` is a thin ctypes layer over it.  Importing
this package does not load the library, so the seeded input generators in
``paper_2207_10731_gb300.workloads`` can be used without a GPU.
"""

__all__ = ["binding", "workloads", "build"]

"""SimSD verification hot path on GB300 (sm_103a).

The CUDA library ``libsimsd.so`` (built from ``csrc/``) holds every step of
the verification forward: the temporal-mask metadata, the split-KV
verification attention, the greedy acceptance and the KV commit.  The Python
side (``simsd``) only marshals arguments into its C ABI; ``inputs`` draws the
seeded synthetic workloads.  Submodules are imported on demand so that the
input generator can be used on hosts without a GPU.
"""

__all__ = ["simsd", "inputs", "build"]

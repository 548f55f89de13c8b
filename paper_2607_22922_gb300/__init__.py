"""GB300-native query path of iFVS (arXiv 2607.22922).

``paper_2607_22922_gb300.ifvs`` is the Python binding of the C-ABI library
``libifvs.so`` (argument marshalling only; every step of the query path runs
in the library's CUDA kernels).  ``paper_2607_22922_gb300.synth`` draws
seeded synthetic inputs.  Nothing is imported eagerly so that the input
generator can be used without the CUDA library.
"""
__all__ = ["ifvs", "synth"]

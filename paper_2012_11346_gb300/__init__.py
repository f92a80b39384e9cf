"""libslim: sliced causal linear (Performer) attention on GB300 (sm_103a).

Importing the package loads nothing; libslim.so is loaded on the first call
into paper_2012_11346_gb300.slim.  Build it with
`python -m paper_2012_11346_gb300.build`.
"""
__all__ = ["slim", "workloads", "build"]

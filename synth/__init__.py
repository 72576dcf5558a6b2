"""Seeded synthetic inputs (session traces and live-set records).

This package generates inputs only.  It holds none of the scheduling
method's arithmetic, and both the CPU oracle and the CUDA library consume
what it produces.
"""
from .traces import (Trace, make_trace, tiny_trace, paper_scale_trace, large_pool_trace,
                     bimodal_trace, trace_from_turns, geometric_turns, save_utr, load_utr,
                     GAP_MIX_CODING, GAP_MIX_GENERAL, GAP_MIX_CONFIG0)
from .records import Records, make_records

__all__ = ["Trace", "make_trace", "tiny_trace", "paper_scale_trace", "large_pool_trace",
           "bimodal_trace", "trace_from_turns", "geometric_turns", "save_utr", "load_utr",
           "GAP_MIX_CODING", "GAP_MIX_GENERAL", "GAP_MIX_CONFIG0", "Records", "make_records"]

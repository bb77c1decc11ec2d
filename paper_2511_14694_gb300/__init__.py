"""FOCUS compressed-context attention on GB300 (arXiv 2511.14694).

The compute path is the C-ABI library ``libfocus.so`` (hand-written sm_103a
CUDA); ``paper_2511_14694_gb300.focus`` is its thin ctypes binding.
"""

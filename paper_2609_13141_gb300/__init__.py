"""GB300-native SAS attention forward (arXiv 2609.13141).

The compute path lives in the C-ABI library built from ``csrc/``; the
Python binding in :mod:`paper_2609_13141_gb300.sas` only marshals arguments.
"""

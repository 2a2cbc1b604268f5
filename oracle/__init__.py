"""fp64 CPU oracle for the GRPO log-prob / policy-loss path (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline / reference
legs import this package; the product package never does.
"""

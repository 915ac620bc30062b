"""TEST INFRASTRUCTURE: the float64 CPU oracle of the policy-loss path.

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
legs may import this package. It shares no code with the CUDA library.
"""

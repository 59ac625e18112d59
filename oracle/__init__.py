"""CPU oracle for the budget-routed decode step — test infrastructure only.

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
legs may import anything under oracle/.  The CUDA path never does.
"""

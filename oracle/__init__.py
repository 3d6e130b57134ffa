"""CPU oracle of the SJD-PAC verify-and-draft step (test infrastructure).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline and
reference legs may import this package; the product path never does.
"""

"""CPU oracle for the MAP pruning path: test infrastructure, never product code.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline arm may import it.
"""

"""CPU oracle for the MXINT mixed-precision linear layer -- test infrastructure only.

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
legs may import this package.  See mxo.c for the definitions it follows.
"""

"""CPU oracle for the VisionPulse decode step: test infrastructure only.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg and
reference arm may import this package.  The library never does.
"""

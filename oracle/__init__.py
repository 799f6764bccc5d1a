"""Test infrastructure: the plain CPU oracle of the T-LoopFormer decode step.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline legs may
import anything from this package.
"""

"""CPU oracle of the Jacobi-decoding hot path (TEST INFRASTRUCTURE ONLY).

Plain fp64 C (jf_oracle.c) behind ctypes (oracle.py) and the decoding loops (jacobi.py).
Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may import it.
"""

"""Oracle (test infrastructure only): a plain fp64 CPU decoder with greedy AR,
Jacobi (refill and shrink) and vanilla Jacobi decoding.  Only tests/,
__graft_entry__.smoke() and bench.py's CPU-baseline leg may import it."""

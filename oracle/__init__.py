"""CPU oracle of the SCM hot path -- TEST INFRASTRUCTURE ONLY.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may import this
package. It shares no code with the CUDA path: `guards` restates Algorithm 1 and the
guard predicates in plain Python; `layer` wraps plain C loops (layer_math.c) for the
decoder-layer math in fp64.
"""

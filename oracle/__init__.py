"""Oracle package -- TEST INFRASTRUCTURE ONLY.

A plain CPU restatement of what the batched-softmax hot path computes
(softmax_oracle.c, double precision) and of the paper's scheduling steps
(schedule_oracle.py).  Only tests/, __graft_entry__.smoke() and bench.py's
CPU-baseline leg may import it; the product path never does.  It imports
nothing from the CUDA package.
"""

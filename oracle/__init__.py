"""fp64 CPU oracle for the offloaded composite regions.

TEST INFRASTRUCTURE.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  It shares no code
with the CUDA path and never imports the product package except its seeded
input module (``paper_2105_03215_gb300.inputs``), which holds no operator
arithmetic.

* ``byoc_oracle.c``   direct-loop fp64 operators (conv2d with groups, dense,
                      bias_add, batch_norm, relu, relu6, gelu, add, pools)
* ``ops``             ctypes wrappers of those loops
* ``graph``           evaluation of an op list node by node (unfolded chain:
                      batch norm is never folded, weights never rounded)
* ``partition_ref``   an independent reference of the partitioning
                      bookkeeping (union-find regions, brute-force maximality)
"""

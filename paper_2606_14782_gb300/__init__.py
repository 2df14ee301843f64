"""GB300-native BACON KV-cache compression (Boundary Attention CalibratiON).

The compute path is the C-ABI library ``libbacon.so`` built from ``csrc/``
for sm_103a; ``bacon`` is its thin Python binding.
"""

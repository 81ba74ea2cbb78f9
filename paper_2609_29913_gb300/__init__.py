"""GB300-native decode attention over a block-wise low-rank KV prefix (MILO).

The compute path is the C-ABI library ``libmilo`` (hand-written sm_103a
kernels) reached through :mod:`paper_2609_29913_gb300.milo`."""

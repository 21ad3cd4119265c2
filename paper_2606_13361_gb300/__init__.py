"""GB300-native KV-cache reuse attention ("Can I Buy Your KV Cache?",
arXiv 2606.13361): C-ABI library libkvr (csrc/, include/kvr.h) and its thin
Python binding (kvr.py).  ``inputs`` holds the seeded synthetic workloads.

The binding is imported lazily (``from paper_2606_13361_gb300 import kvr``) so
that the input generators import without the compiled library."""

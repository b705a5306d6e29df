"""LM-GC encode hot path on GB300 (sm_103a): C-ABI library liblmgc.so and its Python binding."""

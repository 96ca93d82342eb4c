"""fp64 CPU oracle of the MoE expert layer (``moe_oracle``) and of the sequential
collaborative training built on it (``train_oracle``, Alg. 1 on a toy block).

TEST INFRASTRUCTURE ONLY: imported by tests/, ``__graft_entry__.smoke()`` and the
CPU-baseline legs of ``bench.py``, never by the product path. It shares no code
with the CUDA library and imports nothing from it.
"""

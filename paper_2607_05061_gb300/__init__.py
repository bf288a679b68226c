"""KVpop decode hot path on GB300 (sm_103a): C-ABI CUDA library + thin binding.

``paper_2607_05061_gb300.kvpop`` loads ``libkvpop.so`` (build it with
``python -m paper_2607_05061_gb300.build``) and exposes the ABI calls under
their C names plus the ``KVpopCache`` convenience class.
"""

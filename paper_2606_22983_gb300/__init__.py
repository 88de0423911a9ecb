"""GB300-native interaction-aware KV swap path (liblv + thin Python binding).

``build()`` compiles liblv.so for sm_103a in-tree.  The binding
(``paper_2606_22983_gb300.lv``), the pool wrapper (``.pool.KVPool``) and the KV
manager (``.manager.KVManager``) load the compiled library when imported and
fail loudly if it is missing: there is no CPU path.
"""
from ._build import build, LIB  # noqa: F401

"""GB300-native TGV-KV eviction step (score -> budget -> select -> compact).

The computation lives in ``libtgvkv.so`` (hand-written CUDA for sm_103a) behind
the C ABI of ``include/tgvkv.h``; ``api`` is its Python binding.  ``synth``
draws seeded synthetic workloads.  The library is loaded on first use and a
missing build raises; there is no CPU fallback.
"""
from . import synth  # noqa: F401

STATUS_BITS = {
    0x01: "TEXT_POS", 0x02: "VISION_COUNT", 0x04: "BUDGET", 0x08: "INDEX",
    0x10: "COUNT", 0x20: "TIMEOUT", 0x40: "WEIGHT",
}


def __getattr__(name):
    # the binding imports torch; load it lazily so that ``synth`` stays light
    if name == "api":
        import importlib
        return importlib.import_module(".api", __name__)
    raise AttributeError(name)

"""GB300-native joint evaluator (FlashEvaluator, arXiv 2603.02565).

The evaluation runs in libfe.so (hand-written sm_103a CUDA behind a C-ABI,
declared in include/fe.h); `binding.Evaluator` is its Python face.  Build the
library with `paper_2603_02565_gb300.build.build()`.
"""

__all__ = ["Evaluator", "FeError", "load_library"]


def __getattr__(name):
    if name in __all__:
        from . import binding
        return getattr(binding, name)
    raise AttributeError(name)

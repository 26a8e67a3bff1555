"""GB300-native WaveZip video-token condensation (arXiv 2607.23265).

The compute path is the CUDA library libwavezip.so (C ABI in include/wavezip.h);
this package holds its build script (``build``) and a thin ctypes binding
(``wavezip``).  The binding's names are re-exported lazily so that the build
module imports without the library; touching any binding name loads it and
fails loudly if it has not been built.
"""

import importlib


def __getattr__(name):
    if name in ("build", "wavezip"):
        return importlib.import_module(f".{name}", __name__)
    mod = importlib.import_module(".wavezip", __name__)
    try:
        return getattr(mod, name)
    except AttributeError:
        raise AttributeError(f"module {__name__!r} has no attribute {name!r}") from None

"""GB300-native decode-step weight streaming (A-IO, arxiv 2604.09752).

Submodules:
  aio       -- ctypes binding of libaio.so (include/aio.h), same names as the C ABI
  workload  -- device-resident synthetic decode-step workloads (torch for memory only)
  build     -- nvcc build of libaio.so for sm_103a

``aio`` is imported lazily so that ``build`` works before libaio.so exists.
"""


def __getattr__(name):
    if name in ("aio", "workload"):
        import importlib
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)

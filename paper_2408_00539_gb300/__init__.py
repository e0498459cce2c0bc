"""ISM attention on GB300: Python binding of the libism C ABI.

``paper_2408_00539_gb300.ism`` holds the binding (fwd, bwd, prefill_append,
tile_map); ``paper_2408_00539_gb300.workloads`` the seeded synthetic inputs.
The binding is imported lazily so that the workload generator can be used
without a GPU.
"""


def __getattr__(name):
    if name in ("ism", "build", "workloads"):
        import importlib
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)

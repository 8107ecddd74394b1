"""Per-process cache of seeded workload parameters and inputs for the tests."""
import functools

import synth


@functools.lru_cache(maxsize=None)
def params(name: str):
    wl = synth.workload(name)
    return synth.make_params(wl.layers, wl.seed)


@functools.lru_cache(maxsize=None)
def inputs(name: str, batch: int, first: int = 0):
    return synth.make_input(synth.workload(name), batch=batch, first=first)

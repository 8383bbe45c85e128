"""Helpers for the mutant checks of the oracles (CPU): build a copy of an
oracle module with one source fragment replaced, and run a pin module's
test functions (with their parametrizations) against that copy."""
from __future__ import annotations

import inspect
import types


def mutant(module, src_from: str, src_to: str, name: str = "oracle_mutant"):
    """A fresh module from `module`'s source with the first `src_from` replaced."""
    src = inspect.getsource(module)
    assert src_from in src, f"mutation site not found: {src_from[:60]!r}"
    mod = types.ModuleType(name)
    mod.__dict__["__name__"] = name
    exec(compile(src.replace(src_from, src_to, 1), name, "exec"), mod.__dict__)
    return mod


def pins(pin_module):
    return [(n, f) for n, f in inspect.getmembers(pin_module, inspect.isfunction) if n.startswith("test_")]


def call(fn):
    """Runs a pin, once per parameter set of its (single) parametrize mark."""
    params = [m for m in getattr(fn, "pytestmark", []) if m.name == "parametrize"]
    if not params:
        fn()
        return
    names = [s.strip() for s in params[0].args[0].split(",")]
    for vals in params[0].args[1]:
        vals = vals if isinstance(vals, tuple) else (vals,)
        fn(**dict(zip(names, vals)))


def caught_by(pin_module) -> list[str]:
    """Names of the pins that fail (an assertion, or any error a plausible
    mistake raises) against whatever the pin module currently imports."""
    out = []
    for name, fn in pins(pin_module):
        try:
            call(fn)
        except Exception:  # noqa: BLE001 -- a crash on a mutant is a catch
            out.append(name)
    return out

"""GB300-native (sm_103a) VMamba SS2D selective scan: the full-channel scan and
the VMeanba channel-mean scan (arXiv 2412.16602), behind the C ABI of
``libvmb.so`` (include/vmb.h).

``paper_2412_16602_gb300.vmb`` is the Python binding.  Its names are also
available here; the first access loads ``libvmb.so`` and raises ImportError
if the library has not been built (there is no fallback path)."""
import importlib

__all__ = ["vmb"]


def __getattr__(name):
    if name.startswith("__"):
        raise AttributeError(name)
    if name.startswith("_") or name == "vmb":  # submodules: _build, vmb
        try:
            return importlib.import_module("." + name, __name__)
        except ModuleNotFoundError:
            raise AttributeError(f"module {__name__!r} has no attribute {name!r}") from None
    mod = importlib.import_module(".vmb", __name__)
    try:
        return getattr(mod, name)
    except AttributeError:
        raise AttributeError(f"module {__name__!r} has no attribute {name!r}") from None

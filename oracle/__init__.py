"""fp64 CPU oracle for SelKV (test infrastructure only; see selkv_oracle's header)."""
from .selkv_oracle import *  # noqa: F401,F403
from . import selkv_oracle  # noqa: F401

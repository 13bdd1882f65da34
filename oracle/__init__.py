"""CPU oracle package (test infrastructure only; the library never imports it)."""
from .outlets_oracle import *  # noqa: F401,F403

"""CPU oracle of the BRISK-DLM decode tail: test infrastructure only (see brisk_oracle)."""
from .brisk_oracle import *  # noqa: F401,F403

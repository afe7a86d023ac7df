"""CPU oracle of the TaskPress compression path (test infrastructure only)."""
from . import taskpress_oracle  # noqa: F401

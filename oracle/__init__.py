"""fp64 CPU oracle for EG-MLA decode: test infrastructure, never used by the library."""
from .egmla_oracle import *  # noqa: F401,F403

"""CPU oracle of the ExTernD method (fp64, numpy). Test infrastructure: never imported by the product path."""
from .externd_oracle import *  # noqa: F401,F403
from .externd_next import *  # noqa: F401,F403

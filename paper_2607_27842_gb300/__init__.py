"""GB300 (sm_103a) implementation of the FeatFix cached diffusion-transformer
denoising path: a C-ABI CUDA library (include/featfix.h) and its Python
binding.  ``featfix`` is the binding; ``synthetic`` generates seeded inputs
shaped like the paper's backbones."""

from . import featfix  # noqa: F401

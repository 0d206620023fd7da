// Loop-kernel instantiations for shapes 2, 3 of evo_shapes.h (one translation
// unit per group so that the build compiles them in parallel).
#include "evo_loop.cuh"
#include "evo_shapes.h"

namespace evo {

EVO_SHAPE_DEF(2, __nv_bfloat16, 256, 4, 16, 8, 1, 2, 32768, 4)
EVO_SHAPE_DEF(3, __nv_bfloat16, 256, 4, 16, 4, 1, 2, 32768, 4)

}  // namespace evo

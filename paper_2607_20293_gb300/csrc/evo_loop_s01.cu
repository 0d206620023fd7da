// Loop-kernel instantiations for shapes 0, 1 of evo_shapes.h (one translation
// unit per group so that the build compiles them in parallel).
#include "evo_loop.cuh"
#include "evo_shapes.h"

namespace evo {

EVO_SHAPE_DEF(0, __nv_bfloat16, 256, 4, 16, 16, 1, 2, 32768, 4)
EVO_SHAPE_DEF(1, __nv_bfloat16, 256, 4, 16, 16, 2, 2, 32768, 2)

}  // namespace evo

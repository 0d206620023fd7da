// Loop-kernel instantiations for shapes 4, 5 of evo_shapes.h (one translation
// unit per group so that the build compiles them in parallel).
#include "evo_loop.cuh"
#include "evo_shapes.h"

namespace evo {

EVO_SHAPE_DEF(4, __nv_bfloat16, 512, 8, 32, 16, 1, 2, 16384, 2)
EVO_SHAPE_DEF(5, __nv_bfloat16, 64, 2, 8, 4, 1, 2, 32768, 4)

}  // namespace evo

// Loop-kernel instantiations for shapes 6, 7, 8 of evo_shapes.h (one translation
// unit per group so that the build compiles them in parallel).
#include "evo_loop.cuh"
#include "evo_shapes.h"

namespace evo {

EVO_SHAPE_DEF(6, float, 64, 2, 8, 2, 1, 4, 32768, 4)
EVO_SHAPE_DEF(7, float, 64, 2, 8, 4, 1, 4, 32768, 4)
EVO_SHAPE_DEF(8, float, 64, 2, 8, 8, 1, 4, 32768, 4)

}  // namespace evo

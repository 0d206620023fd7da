// Loop-kernel instantiations for shapes 6, 7, 8 of evo_shapes.h (one translation
// unit per group so that the build compiles them in parallel).
#include "evo_loop.cuh"
#include "evo_shapes.h"

namespace evo {

EVO_SHAPE_DEF_ID(6)
EVO_SHAPE_DEF_ID(7)
EVO_SHAPE_DEF_ID(8)

}  // namespace evo

// Loop-kernel instantiations for shapes 0, 1 of evo_shapes.h (one translation
// unit per group so that the build compiles them in parallel).
#include "evo_loop.cuh"
#include "evo_shapes.h"

namespace evo {

EVO_SHAPE_DEF_ID(0)
EVO_SHAPE_DEF_ID(1)

}  // namespace evo

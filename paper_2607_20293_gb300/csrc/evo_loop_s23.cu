// Loop-kernel instantiations for shapes 2, 3 of evo_shapes.h (one translation
// unit per group so that the build compiles them in parallel).
#include "evo_loop.cuh"
#include "evo_shapes.h"

namespace evo {

EVO_SHAPE_DEF_ID(2)
EVO_SHAPE_DEF_ID(3)

}  // namespace evo

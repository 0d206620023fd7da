// Loop-kernel instantiations for shapes 4, 5 of evo_shapes.h (one translation
// unit per group so that the build compiles them in parallel).
#include "evo_loop.cuh"
#include "evo_shapes.h"

namespace evo {

EVO_SHAPE_DEF_ID(4)
EVO_SHAPE_DEF_ID(5)

}  // namespace evo

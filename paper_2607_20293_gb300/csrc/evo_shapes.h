// Compiled loop-kernel shapes: id, operand type, n_emb, heads, horizon,
// cluster size, samples per job, operand bytes, ring slot bytes, ring slots.
// Every workload of this library maps to one of these; other shapes are
// rejected at evo_create (EVO_ERR_UNSUPPORTED).
#pragma once

#define EVO_SHAPES(X)                                           \
  X(0, __nv_bfloat16, 256, 4, 16, 16, 1, 2, 32768, 4)          \
  X(1, __nv_bfloat16, 256, 4, 16, 16, 2, 2, 32768, 2)          \
  X(2, __nv_bfloat16, 256, 4, 16, 8, 1, 2, 32768, 4)           \
  X(3, __nv_bfloat16, 256, 4, 16, 4, 1, 2, 24576, 3)           \
  X(4, __nv_bfloat16, 512, 8, 32, 16, 1, 2, 16384, 2)          \
  X(5, __nv_bfloat16, 64, 2, 8, 4, 1, 2, 32768, 4)             \
  X(6, float, 64, 2, 8, 2, 1, 4, 32768, 4)                     \
  X(7, float, 64, 2, 8, 4, 1, 4, 32768, 4)                     \
  X(8, float, 64, 2, 8, 8, 1, 4, 32768, 4)

#define EVO_SHAPE_DECL(id, T, E, NH, H, C, G, ES, SLOT, NSLOT)                   \
  cudaError_t shape_prepare_##id(int smem_bytes, int* max_clusters);            \
  cudaError_t shape_launch_##id(const JobParams& p, int n_clusters, cudaStream_t s);

// Parameters of shape `id` as types (defined where the loop kernel is visible)
#define EVO_SHAPE_SPEC(id, T_, E, NH, H, C, G, ES, SLOT, NSLOT) \
  template <>                                                  \
  struct ShapeOf<id> {                                         \
    using T = T_;                                              \
    using S = Shape<E, NH, H, C, G, ES, SLOT, NSLOT>;          \
  };

// Host entry points of shape `id`; a translation unit names the ids it
// instantiates, the parameters come from the table above
#define EVO_SHAPE_DEF_ID(id)                                                                      \
  cudaError_t shape_prepare_##id(int smem_bytes, int* max_clusters) {                            \
    return shape_prepare<ShapeOf<id>::T, ShapeOf<id>::S>(smem_bytes, max_clusters);               \
  }                                                                                              \
  cudaError_t shape_launch_##id(const JobParams& p, int n_clusters, cudaStream_t s) {             \
    return shape_launch<ShapeOf<id>::T, ShapeOf<id>::S>(p, n_clusters, s);                        \
  }

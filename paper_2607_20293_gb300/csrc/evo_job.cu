// Small kernels of the path -- the condition tokens' keys/values, the
// lattice check and the population deviation -- plus the host-side
// shared-memory plan of the loop kernel and the dispatch over its compiled
// shapes (the loop kernel itself is in evo_loop.cuh).

#include <algorithm>

#include "evo_ptx.cuh"
#include "evo_tc.cuh"
#include "evo_shapes.h"

namespace evo {

EVO_SHAPES(EVO_SHAPE_DECL)

// ---------------------------------------------------------------------------
// condition path: keys/values of the memory tokens for every layer.  Tokens are
// the timestep token of every loop step (once per handle) and the observation
// tokens of every sample (once per call).  token -> embedding -> MLP E -> 4E
// (Mish) -> E -> per-layer [k | v] = m W_kv + b_kv.  Each matmul is one
// column-parallel launch over all tokens.
// ---------------------------------------------------------------------------

// X[tok][E]: mode 0 = observation token j = tok % n_obs of sample tok / n_obs
// (obs W_obs + b_obs + cond_pos[1+j]); mode 1 = timestep token of loop step tok
// (sinusoidal embedding of the diffusion timestep + cond_pos[0]).
__global__ void cond_embed_kernel(const float* w, const int* wo, const float* obs, const float* kstep, int n_obs, int D,
                                  int E, int mode, float* X) {
  const int tok = blockIdx.x;
  float* x = X + (long long)tok * E;
  if (mode == 0) {
    const int j = tok % n_obs;
    const float* o = obs + (long long)tok * D;
    for (int e = threadIdx.x; e < E; e += blockDim.x) {
      float a = 0.f;
      for (int d = 0; d < D; ++d) a = fmaf(o[d], w[wo[W_OBS_W] + (long long)d * E + e], a);
      x[e] = a + w[wo[W_OBS_B] + e] + w[wo[W_COND_POS] + (1 + j) * E + e];
    }
  } else {
    const double k = (double)kstep[tok];
    const int half = E / 2;
    for (int i = threadIdx.x; i < half; i += blockDim.x) {
      const double f = exp(-log(10000.0) * (double)i / (double)(half - 1));
      x[i] = (float)sin(k * f) + w[wo[W_COND_POS] + i];
      x[half + i] = (float)cos(k * f) + w[wo[W_COND_POS] + half + i];
    }
  }
}

constexpr int GV_TOK = 8;    // tokens per block
constexpr int GV_COLS = 32;  // output columns per block (one per lane)
constexpr int GV_KG = 8;     // K split over the block's 8 warps

// Y[tok][c] = act(X[tok] . W[:, c] + bias[c]) for c < ncols.  Column c lies in
// segment c / seg_cols: W = W0 + seg * seg_stride (row stride ldw), bias =
// b0 + seg * bseg_stride.  act 1 = Mish.
__global__ void __launch_bounds__(256) gemv_cols_kernel(const float* X, int ntok, int K, int ncols, const float* W0,
                                                        long long seg_stride, int seg_cols, int ldw, const float* b0,
                                                        long long bseg_stride, float* Y, int act) {
  extern __shared__ float xs[];                 // [GV_TOK][K], then [GV_KG][GV_TOK][GV_COLS]
  float* red = xs + GV_TOK * K;
  const int t0 = blockIdx.y * GV_TOK;
  const int nt = min(GV_TOK, ntok - t0);
  for (int v = threadIdx.x; v < nt * K; v += blockDim.x) xs[v] = X[(long long)t0 * K + v];
  __syncthreads();
  const int lane = threadIdx.x & 31, kg = threadIdx.x >> 5;
  const int c = blockIdx.x * GV_COLS + lane;
  float acc[GV_TOK];
#pragma unroll
  for (int i = 0; i < GV_TOK; ++i) acc[i] = 0.f;
  if (c < ncols) {
    const int seg = c / seg_cols, cc = c - seg * seg_cols;
    const float* wcol = W0 + seg * seg_stride + cc;
    const int kper = (K + GV_KG - 1) / GV_KG;
    const int k0 = kg * kper, k1 = min(K, k0 + kper);
#pragma unroll 4
    for (int k = k0; k < k1; ++k) {
      const float wk = wcol[(long long)k * ldw];
#pragma unroll
      for (int i = 0; i < GV_TOK; ++i) acc[i] = fmaf(xs[i * K + k], wk, acc[i]);
    }
  }
#pragma unroll
  for (int i = 0; i < GV_TOK; ++i) red[(kg * GV_TOK + i) * GV_COLS + lane] = acc[i];
  __syncthreads();
  // warp kg finishes token kg of the block
  if (kg < nt && c < ncols) {
    float v = 0.f;
#pragma unroll
    for (int g = 0; g < GV_KG; ++g) v += red[(g * GV_TOK + kg) * GV_COLS + lane];
    const int seg = c / seg_cols, cc = c - seg * seg_cols;
    v += b0[seg * bseg_stride + cc];
    if (act) v = mish(v);
    Y[(long long)(t0 + kg) * ncols + c] = v;
  }
}

// tokens [ntok][E] -> keys/values kv[ntok][L][2E]; scratch: ntok * 5E floats
static cudaError_t cond_tokens_to_kv(const float* w, const int* wo_dev, const int* wo, int L, int E, int ntok,
                                     const float* X, float* scratch, float* kv, cudaStream_t s) {
  float* Hd = scratch;                          // [ntok][4E]
  float* Md = scratch + (size_t)ntok * 4 * E;   // [ntok][E]
  const int ty = (ntok + GV_TOK - 1) / GV_TOK;
  auto smem = [](int K) { return (size_t)(GV_TOK * K + GV_KG * GV_TOK * GV_COLS) * sizeof(float); };
  if (smem(4 * E) > 48 * 1024) {
    // above the default dynamic shared memory limit (n_emb > 256)
    const cudaError_t e = cudaFuncSetAttribute(gemv_cols_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)smem(4 * E));
    if (e != cudaSuccess) return e;
  }
  gemv_cols_kernel<<<dim3((4 * E + GV_COLS - 1) / GV_COLS, ty), 256, smem(E), s>>>(
      X, ntok, E, 4 * E, w + wo[W_CM_W1], 0, 4 * E, 4 * E, w + wo[W_CM_B1], 0, Hd, 1);
  gemv_cols_kernel<<<dim3((E + GV_COLS - 1) / GV_COLS, ty), 256, smem(4 * E), s>>>(
      Hd, ntok, 4 * E, E, w + wo[W_CM_W2], 0, E, E, w + wo[W_CM_B2], 0, Md, 0);
  gemv_cols_kernel<<<dim3((L * 2 * E + GV_COLS - 1) / GV_COLS, ty), 256, smem(E), s>>>(
      Md, ntok, E, L * 2 * E, w + wo[W_LAYER0] + wo[WL_CA_WKV], wo[W_LAYER_STRIDE], 2 * E, 2 * E,
      w + wo[W_LAYER0] + wo[WL_CA_BKV], wo[W_LAYER_STRIDE], kv, 0);
  (void)wo_dev;
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// condition path for a few tokens (bf16 models): every weight byte is read once
// per call, so the three matmuls are spread over many blocks.  Block (g, kb, z)
// takes columns g*256 .. +256 and rows kb*CK .. +CK of W (bf16, [K][N]) for the
// tokens z*8 .. +8; warp w takes rows kb*CK + w, + 8, ..., lane l columns
// 8l .. 8l+7 (one 16-byte load per row).  The block's partial sums go to
// part[z][kb][t][N]; the last block of a column group (a counter, reset by that
// block) adds the KB partials in order, adds the bias, applies the activation
// and writes Y.  Stage 0 builds its input rows itself: the observation token
// embedding obs W_obs + b_obs + cond_pos[1 + j].
// ---------------------------------------------------------------------------

constexpr int CG_COLS = 256, CG_TOK = 8, CG_ROWS = 16;   // columns per block, tokens per block, rows per block

struct CondGemv {
  const float* X;            // [ntok][K] (stage 0: null, obs below)
  const float* obs;          // stage 0: [ntok][D]
  const float* w_obs;        // stage 0: [D][K] fp32, + b_obs [K], cond_pos [1 + n_obs][K]
  const float* b_obs;
  const float* pos;
  int D, n_obs;
  int ntok, K, N;
  const __nv_bfloat16* W;    // [K][N]
  const float* bias;         // [N]
  float* Y;                  // [ntok][N]
  float* part;               // [ceil(ntok/8)][K/16][8][N]
  unsigned* count;           // [ceil(ntok/8)][N/256]
  int act;                   // 1 = Mish
};

__global__ void __launch_bounds__(256) cond_gemv_kernel(const CondGemv a) {
  __shared__ float xs[CG_TOK][CG_ROWS];
  __shared__ __align__(16) float red[8][CG_COLS];
  __shared__ int last;
  const int g = blockIdx.x, kb = blockIdx.y, z = blockIdx.z, KB = gridDim.y;
  const int t0 = z * CG_TOK, nt = min(CG_TOK, a.ntok - t0), k0 = kb * CG_ROWS;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // the next stage may launch now; this one touches memory only after the
  // previous stage (its input, the shared partial sums) has completed
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if (tid < CG_TOK * CG_ROWS) {
    const int t = tid / CG_ROWS, r = tid % CG_ROWS, k = k0 + r;
    float v = 0.f;
    if (t < nt) {
      if (a.X) {
        v = a.X[(long long)(t0 + t) * a.K + k];
      } else {
        const float* o = a.obs + (long long)(t0 + t) * a.D;
        for (int d = 0; d < a.D; ++d) v = fmaf(o[d], a.w_obs[(long long)d * a.K + k], v);
        v += a.b_obs[k] + a.pos[(1 + (t0 + t) % a.n_obs) * a.K + k];
      }
    }
    xs[t][r] = v;
  }
  __syncthreads();
  float acc[CG_TOK][8];
#pragma unroll
  for (int t = 0; t < CG_TOK; ++t)
#pragma unroll
    for (int c = 0; c < 8; ++c) acc[t][c] = 0.f;
  const __nv_bfloat16* wp = a.W + (long long)k0 * a.N + g * CG_COLS + lane * 8;
#pragma unroll
  for (int r = warp; r < CG_ROWS; r += 8) {
    const uint4 raw = __ldg(reinterpret_cast<const uint4*>(wp + (long long)r * a.N));
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&raw);
    float w[8];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 f = __bfloat1622float2(h[q]);
      w[2 * q] = f.x;
      w[2 * q + 1] = f.y;
    }
#pragma unroll
    for (int t = 0; t < CG_TOK; ++t) {
      const float xv = xs[t][r];
#pragma unroll
      for (int c = 0; c < 8; ++c) acc[t][c] = fmaf(xv, w[c], acc[t][c]);
    }
  }
  // the block's partial of column tid, token by token: the 8 warps in order
  float* part = a.part + ((long long)z * KB + kb) * CG_TOK * a.N;
  const int n = g * CG_COLS + tid;
#pragma unroll
  for (int t = 0; t < CG_TOK; ++t) {
    if (t < nt) {                                   // block-uniform
      float4* dst = reinterpret_cast<float4*>(&red[warp][lane * 8]);
      dst[0] = make_float4(acc[t][0], acc[t][1], acc[t][2], acc[t][3]);
      dst[1] = make_float4(acc[t][4], acc[t][5], acc[t][6], acc[t][7]);
      __syncthreads();
      float sum = 0.f;
#pragma unroll
      for (int w = 0; w < 8; ++w) sum += red[w][tid];
      part[(long long)t * a.N + n] = sum;
      __syncthreads();
    }
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    unsigned* cnt = a.count + z * gridDim.x + g;
    last = atomicAdd(cnt, 1u) == (unsigned)(KB - 1);
    if (last) *cnt = 0u;                   // ready for the next launch (stream-ordered)
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  const float* p0 = a.part + (long long)z * KB * CG_TOK * a.N;
  for (int t = 0; t < nt; ++t) {
    float v = a.bias[n];
    for (int b = 0; b < KB; ++b) v += __ldcg(p0 + ((long long)b * CG_TOK + t) * a.N + n);
    if (a.act) v = mish(v);
    a.Y[(long long)(t0 + t) * a.N + n] = v;
  }
}

bool cond_fast_ok(int E, int L, long long ntok) {
  return E % CG_COLS == 0 && E % CG_ROWS == 0 && ntok <= 4 * CG_TOK && L * 2 * E % CG_COLS == 0;
}

size_t cond_fast_part_floats(int E, int L, long long ntok) {
  const long long zb = (ntok + CG_TOK - 1) / CG_TOK;
  const long long a = (long long)(4 * E / CG_ROWS) * E, b = (long long)(E / CG_ROWS) * L * 2 * E;
  return (size_t)(zb * CG_TOK * std::max(std::max(a, (long long)(E / CG_ROWS) * 4 * E), b));
}

// w16: [E][4E] | [4E][E] | [E][L*2E] bf16; bkv: [L*2E] fp32; scratch: 5E floats per token
cudaError_t launch_obs_cond_fast(const float* w, const int* wo, const __nv_bfloat16* w16, const float* bkv,
                                 const float* obs, int N, int n_obs, int D, int L, int E, float* scratch,
                                 float* part, unsigned* count, float* kv_obs, cudaStream_t s) {
  const int ntok = N * n_obs, zb = (ntok + CG_TOK - 1) / CG_TOK;
  float* Hd = scratch;                          // [ntok][4E]
  float* Md = scratch + (size_t)ntok * 4 * E;   // [ntok][E]
  CondGemv a{};
  a.ntok = ntok;
  a.part = part;
  a.count = count;
  // stage 0: embedding + E -> 4E, Mish
  a.X = nullptr;
  a.obs = obs;
  a.w_obs = w + wo[W_OBS_W];
  a.b_obs = w + wo[W_OBS_B];
  a.pos = w + wo[W_COND_POS];
  a.D = D;
  a.n_obs = n_obs;
  a.K = E;
  a.N = 4 * E;
  a.W = w16;
  a.bias = w + wo[W_CM_B1];
  a.Y = Hd;
  a.act = 1;
  cond_gemv_kernel<<<dim3(a.N / CG_COLS, a.K / CG_ROWS, zb), 256, 0, s>>>(a);
  // 4E -> E
  a.X = Hd;
  a.K = 4 * E;
  a.N = E;
  a.W = w16 + (size_t)E * 4 * E;
  a.bias = w + wo[W_CM_B2];
  a.Y = Md;
  a.act = 0;
  a.count = count + 256;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.blockDim = dim3(256);
  cfg.stream = s;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(a.N / CG_COLS, a.K / CG_ROWS, zb);
  cudaError_t e = cudaLaunchKernelEx(&cfg, cond_gemv_kernel, a);
  if (e != cudaSuccess) return e;
  // every layer's [k | v]
  a.X = Md;
  a.K = E;
  a.N = L * 2 * E;
  a.W = w16 + (size_t)8 * E * E;
  a.bias = bkv;
  a.Y = kv_obs;
  a.count = count + 512;
  cfg.gridDim = dim3(a.N / CG_COLS, a.K / CG_ROWS, zb);
  e = cudaLaunchKernelEx(&cfg, cond_gemv_kernel, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

__global__ void validate_kernel(const uint8_t* S, long long n, int* err) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
    if (S[i] > 1) atomicOr(err, 1);
}

__global__ void pop_dev_kernel(const float* x, int P, int N_obs, int HA, float* dev) {
  const int pidx = blockIdx.x;
  __shared__ float red[32];
  const float* ref = x + (long long)P * N_obs * HA;
  const float* xp = x + (long long)pidx * N_obs * HA;
  float acc = 0.f;   // sum over n of ||x_pn - x_ref,n||
  for (int n = 0; n < N_obs; ++n) {
    float s = 0.f;
    for (int v = threadIdx.x; v < HA; v += blockDim.x) {
      const float d = xp[(long long)n * HA + v] - ref[(long long)n * HA + v];
      s = fmaf(d, d, s);
    }
    s = group_sum<32>(s);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
      float tot = 0.f;
      for (int w2 = 0; w2 < (int)(blockDim.x >> 5); ++w2) tot += red[w2];
      acc += sqrtf(tot);
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) dev[pidx] = acc / N_obs;
}

// ---------------------------------------------------------------------------
// host-side helpers
// ---------------------------------------------------------------------------

int smem_layout(JobParams& p, int es, int cache_smem) {
  auto al = [](int x, int a) { return (x + a - 1) / a * a; };
  SmemLayout s{};
  int off = 0;
  s.ring = off;
  off += p.nslot * p.slot_bytes;
  // zero-initialised block: ablk .. oc
  s.ablk = off;
  off += al(p.C * p.blk * 4, 128);
  s.rs = off;
  off += al(p.C * p.blk * 4, 128);
  const int xb = p.Mp * p.lda * es;
  const int g1b = p.M * p.ldg1 * 4 > p.Mp * p.ldh * es ? p.M * p.ldg1 * 4 : p.Mp * p.ldh * es;
  s.xln = off;
  off += al(xb > g1b ? xb : g1b, 128);
  // head partials: double-buffered landing blocks of M*npr floats, or one set
  // landing in ablk (block c at c*blk, where a unit's exchanges put c's data)
  if (p.head_sep) {
    s.hblk = off;
    off += al(2 * p.C * p.M * p.npr * 4, 128);
  } else {
    s.hblk = s.ablk;
  }
  s.hsrc = off;
  off += al((p.head_sep ? 2 : 1) * p.M * p.npr * 4, 128);
  s.pb = off;
  off += al(p.M * PLD * 4, 128);
  s.oc = off;
  off += al(p.Mp * p.ldo * es, 128);
  s.ac = off;                                   // end of the zero-initialised block
  off += al(p.M * p.Ec * 4, 128);
  s.acb = off;
  off += al(p.M * p.Ec * 2, 128);
  if (cache_smem) {
    s.cs = off;
    off += al(p.U * p.M * p.Ec * es, 128);
  } else {
    s.cs = -1;
  }
  s.kvs = off;
  off += al(p.kv_slots * p.g * p.Cm * p.kvw * 4, 128);
  s.cst = off;
  off += al((p.A * p.Ec + p.Ec + p.H * p.Ec + 3 * ((p.A + 3) & ~3) + p.A * p.Ec) * 4, 128);
  s.x = off;
  off += al(p.M * p.A * 4, 16);
  s.z = off;
  off += al(p.M * p.A * 4, 16);
  s.stb = off;
  off += al(p.T * 8 * 4, 16);
  s.sch = off;
  off += al(p.T * 8, 16);
  s.psch = off;
  off += al(p.T * 8, 16);
  s.bars = off;
  off += (2 * p.nslot + 5) * 8;
  s.total = al(off, 128);
  p.sm = s;
  return s.total;
}

// ---------------------------------------------------------------------------
// dispatch over the compiled loop-kernel shapes (evo_shapes.h)
// ---------------------------------------------------------------------------

int shape_find(int dtype, int E, int NH, int H, int C, int G, int* slot, int* nslot) {
  struct Row {
    int id, dtype, E, NH, H, C, G, slot, nslot;
  };
#define EVO_SHAPE_ROW(id, T, E_, NH_, H_, C_, G_, ES_, SLOT_, NSLOT_) \
  {id, (ES_ == 2 ? 1 : 0), E_, NH_, H_, C_, G_, SLOT_, NSLOT_},
  static const Row rows[] = {EVO_SHAPES(EVO_SHAPE_ROW)};
#undef EVO_SHAPE_ROW
  for (const Row& r : rows)
    if (r.dtype == dtype && r.E == E && r.NH == NH && r.H == H && r.C == C && r.G == G) {
      *slot = r.slot;
      *nslot = r.nslot;
      return r.id;
    }
  return -1;
}

cudaError_t job_kernel_prepare(int shape, int smem_bytes, int* max_clusters) {
  switch (shape) {
#define EVO_SHAPE_CASE(id, ...) \
  case id:                      \
    return shape_prepare_##id(smem_bytes, max_clusters);
    EVO_SHAPES(EVO_SHAPE_CASE)
#undef EVO_SHAPE_CASE
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_job(int shape, const JobParams& p, int n_clusters, cudaStream_t s) {
  switch (shape) {
#define EVO_SHAPE_CASE(id, ...) \
  case id:                      \
    return shape_launch_##id(p, n_clusters, s);
    EVO_SHAPES(EVO_SHAPE_CASE)
#undef EVO_SHAPE_CASE
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_time_table(const float* w, const int* wo_dev, const int* wo, const float* kstep, int T, int L,
                              int E, float* scratch, float* kv_time, cudaStream_t s) {
  float* X = scratch + (size_t)T * 5 * E;
  cond_embed_kernel<<<T, 256, 0, s>>>(w, wo_dev, nullptr, kstep, 1, 1, E, 1, X);
  return cond_tokens_to_kv(w, wo_dev, wo, L, E, T, X, scratch, kv_time, s);
}

cudaError_t launch_obs_cond(const float* w, const int* wo_dev, const int* wo, const float* obs, int N, int n_obs,
                            int D, int L, int E, float* scratch, float* kv_obs, cudaStream_t s) {
  const int ntok = N * n_obs;
  float* X = scratch + (size_t)ntok * 5 * E;
  cond_embed_kernel<<<ntok, 256, 0, s>>>(w, wo_dev, obs, nullptr, n_obs, D, E, 0, X);
  return cond_tokens_to_kv(w, wo_dev, wo, L, E, ntok, X, scratch, kv_obs, s);
}

// Diagnostic of the device-side failure path: one thread waits on an mbarrier
// that nothing arrives at, through the same bounded-wait helper the loop kernel
// (helper 0) or the tensor-core kernels (helper 1) use.  No cluster, no copy and
// no tensor memory are involved, so giving up leaves nothing in flight.
__global__ void wait_probe_kernel(int helper, long long limit, int* status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (helper == 0) {
      Ctx cx{};
      cx.dead = 0;
      cx.wait_limit = limit;
      wait_parity(smem_u32(&bar), 0u, false, cx, status);
    } else {
      tc::mbar_wait(&bar, 0u, status, limit);
    }
  }
}

cudaError_t launch_wait_probe(int helper, long long limit, int* status, cudaStream_t s) {
  wait_probe_kernel<<<1, 32, 0, s>>>(helper, limit, status);
  return cudaGetLastError();
}

// The feed-forward units' GELU applied to n values: the scalar form of the
// loop kernel (packed = 0) or the packed pair form of the tensor-core GEMM's
// epilogue (packed = 1; an odd last value takes the scalar form).
__global__ void gelu_probe_kernel(const float* x, float* y, long long n, int packed) {
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < (n + 1) / 2; i += stride) {
    if (packed && 2 * i + 1 < n) {
      const float2 r = gelu_as2(make_float2(x[2 * i], x[2 * i + 1]));
      y[2 * i] = r.x;
      y[2 * i + 1] = r.y;
    } else {
      y[2 * i] = gelu_as(x[2 * i]);
      if (2 * i + 1 < n) y[2 * i + 1] = gelu_as(x[2 * i + 1]);
    }
  }
}

cudaError_t launch_gelu_probe(const float* x, float* y, long long n, int packed, cudaStream_t s) {
  if (n > 0)
    gelu_probe_kernel<<<(int)std::min<long long>((n + 511) / 512, 4096), 256, 0, s>>>(x, y, n, packed);
  return cudaGetLastError();
}

cudaError_t launch_validate(const uint8_t* S, long long n, int* err, cudaStream_t s) {
  validate_kernel<<<1, 256, 0, s>>>(S, n, err);
  return cudaGetLastError();
}

cudaError_t launch_pop_dev(const float* x, int P, int N_obs, int HA, float* dev, cudaStream_t s) {
  pop_dev_kernel<<<P, 256, 0, s>>>(x, P, N_obs, HA, dev);
  return cudaGetLastError();
}

}  // namespace evo

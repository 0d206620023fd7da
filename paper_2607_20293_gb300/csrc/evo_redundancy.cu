// Redundancy-aware initialisation (Sec. 3.3): the dissimilarity map of Eq. 6
// from the residual activations of the uncached policy, its MSE / L1 /
// Wasserstein-1 variants, and guided sampling of fixed-budget schedules
// (Eq. 7).
//
// Activations come from evo_denoise_trace with the all-refresh lattice:
// trace [T][U][N][H][E] fp32.  For every unit b and sample r the T activations
// a_{r,b,t} (n = H*E entries each) give the pairwise terms
//   cosine : 1 - <a_t, a_t'> / (|a_t| |a_t'|)      (zero vector: 1)
//   mse    : mean (a_t - a_t')^2
//   l1     : mean |a_t - a_t'|
//   w1     : mean |sort(a_t) - sort(a_t')|          (Wasserstein-1 of the entries)
// and d_{r,b,t} = 1/(T-1) sum_{t' != t} of the term; d_{b,t} = mean over r.
//
// Pair kernel: one block per (b, r).  The T rows are streamed through shared
// memory in chunks of 32 entries; every thread owns register tiles of 4 x 4
// (t, t') pairs and accumulates their dot products or differences over the
// chunks (four FMA-class operations per shared-memory word loaded).  Per-sample maps go to scratch and are averaged in a second pass in
// a fixed order (deterministic).
//
// Guided sampling: one warp per schedule.  The Eq. 7 weights are taken in
// fixed point, q = floor((eps + d/max d)^gamma * 2^40) with IEEE double
// operations that are never contracted, and each draw picks, among the
// positions not yet drawn in index order, the first whose running sum of q
// exceeds rnd mod (sum of the remaining q) (only zero weights left: the
// first position not yet drawn).  All sums are exact 64-bit
// integers, so the schedule does not depend on the order of the warp's scan.

#include <cstdint>
#include <cuda_runtime.h>

#include "evo_internal.h"

namespace evo {

namespace {

constexpr int RM_CH = 64;           // entries per chunk
constexpr int RM_THREADS = 256;
constexpr int RM_MAX_T = 128;

enum { M_COS = 0, M_MSE = 1, M_L1 = 2, M_W1 = 3 };

__host__ __device__ inline int n_pairs(int T) { return T * (T + 1) / 2; }

constexpr int RM_LD = RM_CH + 4;    // shared row stride (floats): 16-byte rows, interleaved tiles hit distinct banks

size_t pair_smem(int T) { return 2 * (size_t)T * RM_LD * sizeof(float) + (size_t)T * T * sizeof(float); }

__device__ __forceinline__ void cp16(float* dst, const float* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src)
               : "memory");
}

template <int METRIC>
__device__ __forceinline__ float pair_op(float x, float y, float acc) {
  if constexpr (METRIC == M_COS) return fmaf(x, y, acc);
  if constexpr (METRIC == M_MSE) {
    const float e = x - y;
    return fmaf(e, e, acc);
  }
  return acc + fabsf(x - y);
}

// One block per (b, r).  The T x T matrix of pair statistics is cut into
// register tiles of 4 x 4 (t, t') pairs; tile (i, j) takes rows
// t in {i, i + Tq, i + 2 Tq, i + 3 Tq} and t' likewise from j (Tq = ceil(T/4)),
// so the float4 loads of neighbouring threads fall in different banks.
// rows: row t of (b, r) starts at base + ((t * U + b) * N + r) * n
template <int METRIC>
__global__ void __launch_bounds__(RM_THREADS, METRIC == M_COS ? 1 : 2) pair_kernel(const float* rows, int T, int U, int N, int n,
                                                          float* dr /* [U][N][T] */) {
  extern __shared__ __align__(16) float rm_smem[];
  float* xb = rm_smem;                                  // 2 x [T][RM_LD]: chunk c in buffer c & 1
  float* G = xb + 2 * T * RM_LD;                        // [T][T]
  const int b = blockIdx.x / N, r = blockIdx.x % N;
  const int Tq = (T + 3) / 4, tiles = Tq * Tq;
  constexpr int TPT = ((RM_MAX_T / 4) * (RM_MAX_T / 4) + RM_THREADS - 1) / RM_THREADS;   // tiles per thread (max)
  float acc[TPT][4][4];
#pragma unroll
  for (int q = 0; q < TPT; ++q)
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[q][a][c] = 0.f;
  // chunk c of every row -> buffer c & 1: 16-byte asynchronous copies when the
  // rows are a multiple of 4 entries, plain loads otherwise (zero-padded tail)
  const int nch = (n + RM_CH - 1) / RM_CH;
  auto load_chunk = [&](int c) {
    float* xs = xb + (c & 1) * T * RM_LD;
    const int c0 = c * RM_CH, w = min(RM_CH, n - c0);
    for (int v = threadIdx.x; v < T * (RM_CH / 4); v += blockDim.x) {
      const int t = v / (RM_CH / 4), k = 4 * (v % (RM_CH / 4));
      const float* src = rows + ((long long)(t * U + b) * N + r) * n + c0 + k;
      float* dst = xs + t * RM_LD + k;
      if (k + 3 < w && (n & 3) == 0) {
        cp16(dst, src);
      } else {
        float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
        if (k < w) f.x = src[0];
        if (k + 1 < w) f.y = src[1];
        if (k + 2 < w) f.z = src[2];
        if (k + 3 < w) f.w = src[3];
        *reinterpret_cast<float4*>(dst) = f;
      }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  load_chunk(0);
  for (int c = 0; c < nch; ++c) {
    if (c + 1 < nch) {
      load_chunk(c + 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();
    const float* xs = xb + (c & 1) * T * RM_LD;
#pragma unroll
    for (int q = 0; q < TPT; ++q) {
      const int tile = threadIdx.x + q * RM_THREADS;
      if (tile < tiles) {
        const int i = tile / Tq, j = tile % Tq;
        int ra[4], rc[4];
#pragma unroll
        for (int a = 0; a < 4; ++a) {
          ra[a] = min(i + a * Tq, T - 1);   // rows beyond T repeat the last row; their results are dropped
          rc[a] = min(j + a * Tq, T - 1);
        }
#pragma unroll 2
        for (int k = 0; k < RM_CH; k += 4) {
          float4 x[4], y[4];
#pragma unroll
          for (int a = 0; a < 4; ++a) {
            x[a] = *reinterpret_cast<const float4*>(xs + ra[a] * RM_LD + k);
            y[a] = *reinterpret_cast<const float4*>(xs + rc[a] * RM_LD + k);
          }
#pragma unroll
          for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int c = 0; c < 4; ++c) {
              float v = acc[q][a][c];
              v = pair_op<METRIC>(x[a].x, y[c].x, v);
              v = pair_op<METRIC>(x[a].y, y[c].y, v);
              v = pair_op<METRIC>(x[a].z, y[c].z, v);
              v = pair_op<METRIC>(x[a].w, y[c].w, v);
              acc[q][a][c] = v;
            }
        }
      }
    }
    __syncthreads();   // buffer c & 1 is refilled with chunk c + 2 next
  }
#pragma unroll
  for (int q = 0; q < TPT; ++q) {
    const int tile = threadIdx.x + q * RM_THREADS;
    if (tile < tiles) {
      const int i = tile / Tq, j = tile % Tq;
#pragma unroll
      for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int t = i + a * Tq, t2 = j + c * Tq;
          if (t < T && t2 < T) G[t * T + t2] = acc[q][a][c];
        }
    }
  }
  __syncthreads();
  for (int t = threadIdx.x; t < T; t += blockDim.x) {
    float s = 0.f;
    for (int t2 = 0; t2 < T; ++t2) {
      if (t2 == t) continue;
      float term;
      if (METRIC == M_COS) {
        const float nn = sqrtf(G[t * T + t]) * sqrtf(G[t2 * T + t2]);
        term = nn == 0.f ? 1.f : 1.f - G[t * T + t2] / nn;
      } else {
        term = G[t * T + t2] / (float)n;
      }
      s += term;
    }
    dr[((long long)b * N + r) * T + t] = s / (float)(T - 1);
  }
}

// d[b][t] = mean over r of dr[b][r][t], summed in order r = 0..N-1
__global__ void mean_kernel(const float* dr, int T, int U, int N, float* d) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= U * T) return;
  const int b = i / T, t = i % T;
  float s = 0.f;
  for (int r = 0; r < N; ++r) s += dr[((long long)b * N + r) * T + t];
  d[i] = s / (float)N;
}

// ascending bitonic sort of each row of n = 2^k entries (one block per row)
__global__ void sort_rows_kernel(const float* in, float* out, int n) {
  extern __shared__ __align__(16) float srt[];
  const float* src = in + (long long)blockIdx.x * n;
  for (int i = threadIdx.x; i < n; i += blockDim.x) srt[i] = src[i];
  __syncthreads();
  for (int k = 2; k <= n; k <<= 1)
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const int l = i ^ j;
        if (l > i) {
          const float a = srt[i], c = srt[l];
          const bool up = (i & k) == 0;
          if ((a > c) == up) {
            srt[i] = c;
            srt[l] = a;
          }
        }
      }
      __syncthreads();
    }
  float* dst = out + (long long)blockIdx.x * n;
  for (int i = threadIdx.x; i < n; i += blockDim.x) dst[i] = srt[i];
}

constexpr int GS_MAX_CELLS = 4096;

// one warp per schedule p
__global__ void __launch_bounds__(32) guided_kernel(const float* d, int cells, int K, float eps, int gamma,
                                                    const unsigned long long* rnd, uint8_t* S) {
  __shared__ long long q[GS_MAX_CELLS];
  __shared__ uint8_t taken[GS_MAX_CELLS];
  const int p = blockIdx.x, lane = threadIdx.x;
  float mx = 0.f;
  for (int i = lane; i < cells; i += 32) mx = fmaxf(mx, d[i]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  const double e = (double)eps, dm = (double)mx;
  for (int i = lane; i < cells; i += 32) {
    const double base = __dadd_rn(e, __ddiv_rn((double)d[i], dm));
    double v = base;
    for (int g = 1; g < gamma; ++g) v = __dmul_rn(v, base);
    q[i] = (long long)floor(__dmul_rn(v, 1099511627776.0));
    taken[i] = 0;
  }
  __syncwarp();
  const int ch = (cells + 31) / 32, lo = lane * ch, hi = min(cells, lo + ch);
  for (int k = 0; k < K; ++k) {
    long long part = 0;
    for (int i = lo; i < hi; ++i)
      if (!taken[i]) part += q[i];
    long long incl = part;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long up = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += up;
    }
    const long long total = __shfl_sync(0xffffffffu, incl, 31);
    int pick = -1;
    if (total == 0) {
      // only zero weights left: the first position not yet drawn
      for (int i = lo; i < hi; ++i)
        if (!taken[i]) {
          pick = i;
          break;
        }
      const unsigned has = __ballot_sync(0xffffffffu, pick >= 0);
      const int sel = __shfl_sync(0xffffffffu, pick, has ? __ffs(has) - 1 : 0);
      if (lane == 0 && sel >= 0) taken[sel] = 1;
      __syncwarp();
      continue;
    }
    const unsigned long long target = rnd[(long long)p * K + k] % (unsigned long long)total;
    const long long excl = incl - part;
    if ((unsigned long long)excl <= target && target < (unsigned long long)incl) {
      long long run = excl;
      for (int i = lo; i < hi; ++i) {
        if (taken[i]) continue;
        run += q[i];
        if ((unsigned long long)run > target) {
          pick = i;
          break;
        }
      }
    }
    const unsigned who = __ballot_sync(0xffffffffu, pick >= 0);
    const int sel = __shfl_sync(0xffffffffu, pick, who ? __ffs(who) - 1 : 0);
    if (lane == 0 && sel >= 0) taken[sel] = 1;
    __syncwarp();
  }
  for (int i = lane; i < cells; i += 32) S[(long long)p * cells + i] = taken[i];
}

}  // namespace

size_t redundancy_scratch_bytes(int T, int U, int N, int n, int metric) {
  size_t b = (size_t)U * N * T * sizeof(float);
  if (metric == M_W1) b += (size_t)T * U * N * n * sizeof(float);
  return b;
}

bool redundancy_shape_ok(int T, int U, int N, int n, int metric) {
  if (T < 2 || T > RM_MAX_T || U <= 0 || N <= 0 || n <= 0 || metric < 0 || metric > M_W1) return false;
  if (metric == M_W1 && ((n & (n - 1)) != 0 || n > 16384)) return false;   // bitonic sort in shared memory
  return true;
}

cudaError_t launch_redundancy(const float* trace, int T, int U, int N, int n, int metric, float* d, void* scratch,
                              cudaStream_t st) {
  float* dr = static_cast<float*>(scratch);
  const float* rows = trace;
  if (metric == M_W1) {
    float* sorted = dr + (size_t)U * N * T;
    const int sm = n * (int)sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(sort_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
    if (e != cudaSuccess) return e;
    sort_rows_kernel<<<T * U * N, 1024, sm, st>>>(trace, sorted, n);
    rows = sorted;
  }
  const int sm = (int)pair_smem(T);
  cudaError_t e = cudaSuccess;
  switch (metric) {
    case M_COS:
      e = cudaFuncSetAttribute(pair_kernel<M_COS>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
      if (e == cudaSuccess) pair_kernel<M_COS><<<U * N, RM_THREADS, sm, st>>>(rows, T, U, N, n, dr);
      break;
    case M_MSE:
      e = cudaFuncSetAttribute(pair_kernel<M_MSE>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
      if (e == cudaSuccess) pair_kernel<M_MSE><<<U * N, RM_THREADS, sm, st>>>(rows, T, U, N, n, dr);
      break;
    default:
      e = cudaFuncSetAttribute(pair_kernel<M_L1>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
      if (e == cudaSuccess) pair_kernel<M_L1><<<U * N, RM_THREADS, sm, st>>>(rows, T, U, N, n, dr);
      break;
  }
  if (e != cudaSuccess) return e;
  mean_kernel<<<(U * T + 255) / 256, 256, 0, st>>>(dr, T, U, N, d);
  return cudaGetLastError();
}

bool guided_shape_ok(int U, int T, int K, int gamma, int P) {
  return U > 0 && T > 0 && U * T <= GS_MAX_CELLS && K >= 0 && K <= U * T && gamma >= 1 && gamma <= 16 && P > 0;
}

cudaError_t launch_guided(const float* d, int U, int T, int K, float eps, int gamma, const uint64_t* rnd, int P,
                          uint8_t* S, cudaStream_t st) {
  guided_kernel<<<P, 32, 0, st>>>(d, U * T, K, eps, gamma, reinterpret_cast<const unsigned long long*>(rnd), S);
  return cudaGetLastError();
}

}  // namespace evo

// Tensor-core GEMM of the batch-wide path: C[rows][N] = A[rows][K] . B[N][K]^T
// on the fifth-generation tensor cores (tcgen05), bf16 operands, fp32
// accumulation in tensor memory, with the epilogues the denoiser needs fused.
//
// Persistent: a CTA per SM walks the BM x BN output tiles (m-major, so
// consecutive tiles reuse the same rows of A from L2), warp-specialised:
//   * warp 0, one lane: TMA producer.  Tiles of A (BM x 64) and B (BN x 64)
//     land in a ring of shared-memory stages with the 128-byte swizzle
//     (cp.async.bulk.tensor + mbarrier transaction counts);
//   * warp 1, one lane: MMA issuer.  Four tcgen05.mma (K = 16 each) per stage
//     into one of two TMEM accumulators of BN columns; tcgen05.commit frees a
//     stage when the MMAs that read it are done, and hands a finished
//     accumulator to the epilogue;
//   * warps 2-9: epilogue.  Warp w reads TMEM lanes (= tile rows) of its
//     quadrant 32 (w % 4) .. +31 and one half of the tile's columns, 32 at a
//     time (tcgen05.ld), applies bias (and GELU / Mish), packs bf16 into its
//     staging rows in shared memory in the 128-byte-swizzled layout, and
//     writes each 32 x 64 block with one tiled bulk store (the thread-per-row
//     layout of the accumulator would scatter every direct store over 32
//     rows), releasing the accumulator as soon as its last columns are in
//     registers.  The residual mode (the output projection of a refreshed
//     unit) stages fp32 r and stores it (a tiled bulk store through tmC, an
//     fp32 map of r, when all 32 rows of a warp refresh the unit) together
//     with the unit's bf16 cache (Eq. 1) for the rows that refresh the unit.
// With two accumulators the epilogue of one tile overlaps the main loop of the
// next.  BN = 256 for large problems, 128 when that leaves SMs idle.
//
// Every wait on an mbarrier is bounded: on expiry the thread records
// ST_TIMEOUT in the status word and carries on, so the kernel always ends.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>

#include "evo_internal.h"

namespace evo {
namespace tc {

constexpr int BM = 128, BK = 64;
constexpr int A_BYTES = BM * BK * 2;
constexpr int EPI_WARPS = 8;                                    // two per TMEM lane quadrant
constexpr int NTHREADS_GEMM = 32 * (2 + EPI_WARPS);             // producer, MMA, epilogue warps

// epilogue staging: per epilogue warp 32 rows x 64 bf16 columns (128-byte rows,
// 16-byte chunks XOR-swizzled by row so that both the thread-per-row writes and
// the warp-per-row reads are free of bank conflicts)
constexpr int EPI_STG_BYTES = EPI_WARPS * 32 * 128;

template <int BN>
struct TileCfg {
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = BN == 256 ? 4 : 6;
  // alignment slack, stages, epilogue staging, barriers
  static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + EPI_STG_BYTES + 256;
  static constexpr int TMEM_COLS = 2 * BN;                                // two accumulators
  // instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both
  // K-major, M = BM, N = BN
  static constexpr uint32_t IDESC =
      (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
};

enum EpiMode { EPI_BF16 = 0, EPI_GELU_BF16 = 1, EPI_RESID = 2, EPI_MISH_BF16 = 3, EPI_F32 = 4 };

struct GemmArgs {
  int K;                      // multiple of BK
  int b_row0;                 // first row of B (its tensor map spans every layer's matrices)
  const float* bias;          // [N] fp32
  __nv_bfloat16* out;         // EPI_BF16 / EPI_GELU_BF16: out[row * ldo + n]
  int ldo;
  float* rout;                // EPI_RESID: the branch output r [rows][ldr] fp32, for refreshing rows
  __nv_bfloat16* cache;       // EPI_RESID: the unit's cache [rows][ldr], <- bf16(r) for refreshing rows
  float* trace;               // EPI_RESID: [rows][ldr] or null: r of refreshing rows (debug trace)
  int ldr;
  float* out32;               // EPI_F32: out32[row * ldo + n]
  const float* rbias;         // bf16 modes, or null: + rbias[(row % rbias_mod) * ldo + n] (a per-row bias)
  int rbias_mod;
  int rows;                   // real rows; rows >= this are padding
  // refresh gate (null: every row refreshes): row -> sample row / H -> lattice
  // (sample / per_sched); refresh = S[lattice * S_stride + srow * T + t]
  const uint8_t* S;
  long long S_stride;
  int srow, T, t, H, per_sched, force;
  int* status;
  long long wait_limit;       // polls before a wait gives up (WAIT_POLLS_DEFAULT)
};

// ---------------------------------------------------------------- PTX wrappers
__device__ __forceinline__ uint32_t su32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init1(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// bounded wait for the phase of `parity` to complete: gives up after `limit`
// polls and records ST_TIMEOUT
__device__ __forceinline__ void mbar_wait(uint64_t* bar, uint32_t parity, int* status, long long limit) {
  const uint32_t a = su32(bar);
  if (mbar_test(a, parity)) return;
  for (long long i = 0; i < limit; ++i) {
    if (mbar_test(a, parity)) return;
    if (i > 64) __nanosleep(32);
  }
  atomicOr(status, ST_TIMEOUT);
}

__device__ __forceinline__ void mbar_arrive1(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(bar)), "r"(bytes) : "memory");
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(su32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(su32(bar))
      : "memory");
}

// tiled bulk store shared -> global (bulk-group completion)
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, int x, int y, const void* src) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(su32(src))
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// the source shared memory of every committed bulk store has been read
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// every committed bulk store has completed
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// this thread's generic-proxy shared-memory writes become visible to the async proxy (bulk copies)
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(slot)), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// Programmatic dependent launch: let the next kernel of the stream start its
// launch now; wait until the previous kernel has finished and its writes are
// visible (a no-op for kernels launched without the attribute).
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor: K-major operand in 128-byte-swizzled rows
// (8-row groups 1024 bytes apart), the layout a SWIZZLE_128B TMA box of 64
// bf16 columns produces.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);      // start address
  d |= (uint64_t)1 << 16;                         // leading byte offset (unused with this swizzle)
  d |= (uint64_t)(1024 >> 4) << 32;               // stride byte offset: next 8-row group
  d |= (uint64_t)1 << 46;                         // descriptor version
  d |= (uint64_t)2 << 61;                         // 128-byte swizzle
  return d;
}

__device__ __forceinline__ void mma_f16(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
          tmem_d),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(bar))
               : "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// the row's lattice refreshes the unit (EPI_RESID writes only such rows)
__device__ __forceinline__ bool row_refreshes(const GemmArgs& g, int row) {
  if (row >= g.rows) return false;
  if (!g.S || (g.force && g.t == 0)) return true;
  const int sample = row / g.H;
  return g.S[(long long)(sample / g.per_sched) * g.S_stride + (long long)g.srow * g.T + g.t] != 0;
}

__device__ __forceinline__ float mish_f(float v) {
  const float sp = v > 20.f ? v : log1pf(expf(v));
  return v * tanhf(sp);
}

// does any row of the tile starting at m0 refresh?  (the same answer in every role)
__device__ __forceinline__ bool tile_live(const GemmArgs& g, int m0) {
  if (m0 >= g.rows) return false;
  if (!g.S || (g.force && g.t == 0)) return true;
  const int last = min(m0 + BM, g.rows) - 1;
  for (int s = m0 / g.H; s <= last / g.H; ++s)
    if (g.S[(long long)(s / g.per_sched) * g.S_stride + (long long)g.srow * g.T + g.t] != 0) return true;
  return false;
}

// (a, b) += (c, d) as one packed add
__device__ __forceinline__ void add2_into(float& a, float& b, float c, float d) {
  const float2 r = add2(make_float2(a, b), make_float2(c, d));
  a = r.x;
  b = r.y;
}

// bias (and GELU / Mish) on 32 accumulator columns n .. n + 31 of this
// thread's row, packed to bf16: pk[q] = columns 8q .. 8q + 7 (registers only,
// so that this work overlaps the bulk store still reading the staging rows)
template <int MODE>
__device__ __forceinline__ void epilogue_values(const GemmArgs& g, int row, int n, float (&v)[32], uint4* pk) {
  const float4* b4 = reinterpret_cast<const float4*>(g.bias + n);
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const float4 bb = __ldg(b4 + q);
    add2_into(v[4 * q], v[4 * q + 1], bb.x, bb.y);
    add2_into(v[4 * q + 2], v[4 * q + 3], bb.z, bb.w);
  }
  if (g.rbias) {
    const float4* r4 = reinterpret_cast<const float4*>(g.rbias + (long long)(row % g.rbias_mod) * g.ldo + n);
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float4 bb = __ldg(r4 + q);
      add2_into(v[4 * q], v[4 * q + 1], bb.x, bb.y);
      add2_into(v[4 * q + 2], v[4 * q + 3], bb.z, bb.w);
    }
  }
  if constexpr (MODE == EPI_GELU_BF16) {
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const float2 y = gelu_as2(make_float2(v[2 * i], v[2 * i + 1]));
      v[2 * i] = y.x;
      v[2 * i + 1] = y.y;
    }
  }
  if constexpr (MODE == EPI_MISH_BF16) {
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = mish_f(v[i]);
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint32_t* pw = reinterpret_cast<uint32_t*>(&pk[q]);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      __nv_bfloat162 h2 = __floats2bfloat162_rn(v[8 * q + 2 * j], v[8 * q + 2 * j + 1]);
      pw[j] = *reinterpret_cast<uint32_t*>(&h2);
    }
  }
}

// EPI_RESID, one chunk of 32 columns n .. n + 31: r = acc + bias goes to the
// warp's staging rows (fp32, thread = row, the 128-byte-swizzled layout of a
// 32 x 32 fp32 box), then for the rows whose lattice refreshes the unit (bit r
// of rmask) r is stored -- by one tiled bulk store through tmR when all 32 rows
// refresh (and no trace is taken), else by the warp (eight lanes per row, 16
// bytes each) -- and c_b <- bf16(r) (Eq. 1) by the warp (four lanes per row,
// eight values each), reading the staging rows alongside the bulk store.  The
// row walk that follows adds r to the residual stream.
__device__ __forceinline__ void epilogue_resid(const GemmArgs& g, const CUtensorMap* tmR, int row0, int n,
                                               float (&v)[32], uint8_t* stg, int lane, unsigned rmask) {
  const bool bulk = rmask == 0xffffffffu && !g.trace;
  if (lane == 0) bulk_wait_read();   // the previous chunk's bulk store has left the staging rows
  __syncwarp();
  const float4* b4 = reinterpret_cast<const float4*>(g.bias + n);
  uint8_t* srow = stg + lane * 128;
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const float4 bb = __ldg(b4 + q);
    add2_into(v[4 * q], v[4 * q + 1], bb.x, bb.y);
    add2_into(v[4 * q + 2], v[4 * q + 3], bb.z, bb.w);
    *reinterpret_cast<float4*>(srow + ((q ^ (lane & 7)) << 4)) =
        make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
  }
  if (bulk) fence_async_smem();
  __syncwarp();
  if (bulk) {
    if (lane == 0) {
      tma_store_2d(tmR, n, row0, stg);
      bulk_commit();
    }
  } else {
    const int cc = lane & 7;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = 4 * i + (lane >> 3);
      if ((rmask >> r) & 1u) {
        const float4 val = *reinterpret_cast<const float4*>(stg + r * 128 + ((cc ^ (r & 7)) << 4));
        const long long o = (long long)(row0 + r) * g.ldr + n + 4 * cc;
        *reinterpret_cast<float4*>(g.rout + o) = val;
        if (g.trace) *reinterpret_cast<float4*>(g.trace + o) = val;
      }
    }
  }
  const int cp = lane & 3;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = 8 * i + (lane >> 2);
    if ((rmask >> r) & 1u) {
      const float4 f0 = *reinterpret_cast<const float4*>(stg + r * 128 + (((2 * cp) ^ (r & 7)) << 4));
      const float4 f1 = *reinterpret_cast<const float4*>(stg + r * 128 + (((2 * cp + 1) ^ (r & 7)) << 4));
      __nv_bfloat162 h[4] = {__floats2bfloat162_rn(f0.x, f0.y), __floats2bfloat162_rn(f0.z, f0.w),
                             __floats2bfloat162_rn(f1.x, f1.y), __floats2bfloat162_rn(f1.z, f1.w)};
      // the cache is read again only by later walks: evict-first, r stays in L2 for the next walk
      __stcs(reinterpret_cast<uint4*>(g.cache + (long long)(row0 + r) * g.ldr + n + 8 * cp),
             *reinterpret_cast<const uint4*>(h));
    }
  }
  __syncwarp();
}

// EPI_F32, one chunk of 32 columns: acc + bias staged as fp32 (thread = row),
// then stored row by row (lane = column, 128 contiguous bytes) for rows < rows
__device__ __forceinline__ void epilogue_f32(const GemmArgs& g, int row0, int n, float (&v)[32], uint8_t* stg,
                                             int lane) {
  const float4* b4 = reinterpret_cast<const float4*>(g.bias + n);
  uint8_t* srow = stg + lane * 128;
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const float4 bb = __ldg(b4 + q);
    *reinterpret_cast<float4*>(srow + ((q ^ (lane & 7)) << 4)) =
        make_float4(v[4 * q] + bb.x, v[4 * q + 1] + bb.y, v[4 * q + 2] + bb.z, v[4 * q + 3] + bb.w);
  }
  __syncwarp();
#pragma unroll 8
  for (int r = 0; r < 32; ++r) {
    if (row0 + r >= g.rows) break;
    g.out32[(long long)(row0 + r) * g.ldo + n + lane] =
        *reinterpret_cast<const float*>(stg + r * 128 + (((lane >> 2) ^ (r & 7)) << 4) + (lane & 3) * 4);
  }
  __syncwarp();
}

// the warp has read its last columns of the accumulator (tcgen05.ld waited):
// one arrival of the EPI_WARPS that free it for the next tile's main loop
__device__ __forceinline__ void release_acc(uint64_t* tempty, int lane) {
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive1(tempty);
}

// ---------------------------------------------------------------- the kernel
// Tiles: m_tiles x n_tiles, tile i -> (i / n_tiles, i % n_tiles); CTA c takes
// tiles c, c + gridDim.x, ...
template <int MODE, int BN>
__global__ void __launch_bounds__(NTHREADS_GEMM, 1) gemm_kernel(const __grid_constant__ CUtensorMap tmA,
                                                                const __grid_constant__ CUtensorMap tmB,
                                                                const __grid_constant__ CUtensorMap tmC,
                                                                const GemmArgs g, int m_tiles, int n_tiles) {
  using C = TileCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES + EPI_STG_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tfull = empty + C::STAGES;     // [2]: accumulator ready for the epilogue
  uint64_t* tempty = tfull + 2;            // [2]: accumulator drained by the epilogue
  uint32_t* tslot = reinterpret_cast<uint32_t*>(tempty + 2);
  if (warp == 1) tmem_alloc(tslot, C::TMEM_COLS);
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init1(&full[s], 1);
      mbar_init1(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init1(&tfull[a], 1);
      mbar_init1(&tempty[a], EPI_WARPS);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();                              // A, the residual stream and the lattice come from earlier kernels
  const uint32_t tmem = *tslot;
  const int KB = g.K / BK, total = m_tiles * n_tiles;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t q = 0;
      for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
        const int m0 = (tile / n_tiles) * BM, n0 = (tile % n_tiles) * BN;
        if (!tile_live(g, m0)) continue;
        for (int kb = 0; kb < KB; ++kb, ++q) {
          const int s = q % C::STAGES;
          mbar_wait(&empty[s], ((q / C::STAGES) & 1u) ^ 1u, g.status, g.wait_limit);
          uint8_t* sa = smem + s * C::STAGE_BYTES;
          mbar_expect_tx(&full[s], C::STAGE_BYTES);
          tma_load_2d(sa, &tmA, kb * BK, m0, &full[s]);
          tma_load_2d(sa + A_BYTES, &tmB, kb * BK, g.b_row0 + n0, &full[s]);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      uint32_t q = 0, it = 0;
      for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
        if (!tile_live(g, (tile / n_tiles) * BM)) continue;
        const uint32_t acc = it & 1u;
        mbar_wait(&tempty[acc], ((it >> 1) & 1u) ^ 1u, g.status, g.wait_limit);
        tc_fence_after();
        const uint32_t d = tmem + acc * BN;
        for (int kb = 0; kb < KB; ++kb, ++q) {
          const int s = q % C::STAGES;
          mbar_wait(&full[s], (q / C::STAGES) & 1u, g.status, g.wait_limit);
          tc_fence_after();
          const uint32_t sa = su32(smem + s * C::STAGE_BYTES);
          const uint64_t da = sw128_desc(sa), db = sw128_desc(sa + A_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)   // +32 bytes along K = +2 in the encoded start address
            mma_f16(d, da + 2 * k, db + 2 * k, C::IDESC, (kb | k) != 0);
          mma_commit(&empty[s]);
        }
        mma_commit(&tfull[acc]);
        ++it;
      }
    }
  } else {
    // epilogue warps: TMEM lane quadrant (warp % 4) = tile rows 32 (warp % 4) ..,
    // column half (warp - 2) / 4; 64 columns at a time through the warp's staging
    const int quad = warp & 3, half = (warp - 2) >> 2;
    uint8_t* stg = smem + C::STAGES * C::STAGE_BYTES + (warp - 2) * 32 * 128;
    uint32_t it = 0;
    for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
      const int m0 = (tile / n_tiles) * BM, n0 = (tile % n_tiles) * BN;
      if (!tile_live(g, m0)) continue;
      const uint32_t acc = it & 1u;
      mbar_wait(&tfull[acc], (it >> 1) & 1u, g.status, g.wait_limit);
      tc_fence_after();
      const uint32_t tq = tmem + acc * BN + ((uint32_t)(quad * 32) << 16);   // this warp's TMEM lanes
      if constexpr (MODE == EPI_F32) {
#pragma unroll 1
        for (int c = half * (BN / 64); c < (half + 1) * (BN / 64); ++c) {
          float v[32];
          tmem_ld32(tq + (uint32_t)(c * 32), v);
          epilogue_f32(g, m0 + quad * 32, n0 + c * 32, v, stg, lane);
        }
      } else if constexpr (MODE == EPI_RESID) {
        const unsigned rmask = __ballot_sync(0xffffffffu, row_refreshes(g, m0 + quad * 32 + lane));
#pragma unroll 1
        for (int c = half * (BN / 64); c < (half + 1) * (BN / 64); ++c) {
          float v[32];
          tmem_ld32(tq + (uint32_t)(c * 32), v);
          if (c + 1 == (half + 1) * (BN / 64)) release_acc(&tempty[acc], lane);   // last columns are in registers
          epilogue_resid(g, &tmC, m0 + quad * 32, n0 + c * 32, v, stg, lane, rmask);
        }
      } else {
        // 32 rows x 64 columns at a time: packed into the staging rows (the
        // layout of a 128-byte-swizzled tile), then one tiled bulk store of the
        // whole block by lane 0 (out of range rows land in the buffer's padding)
#pragma unroll 1
        for (int c = half * (BN / 64); c < (half + 1) * (BN / 64); c += 2) {
          uint4 pk[8];
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            float v[32];
            tmem_ld32(tq + (uint32_t)((c + j) * 32), v);
            epilogue_values<MODE>(g, m0 + quad * 32 + lane, n0 + (c + j) * 32, v, pk + 4 * j);
          }
          if (c + 2 == (half + 1) * (BN / 64)) release_acc(&tempty[acc], lane);
          if (lane == 0) bulk_wait_read();               // the previous block has left the staging rows
          __syncwarp();
          uint8_t* srow = stg + lane * 128;
#pragma unroll
          for (int q = 0; q < 8; ++q) *reinterpret_cast<uint4*>(srow + ((q ^ (lane & 7)) << 4)) = pk[q];
          fence_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&tmC, n0 + c * 32, m0 + quad * 32, stg);
            bulk_commit();
          }
        }
      }
      if constexpr (MODE == EPI_F32) release_acc(&tempty[acc], lane);
      ++it;
    }
  }
  if (warp >= 2 && lane == 0) bulk_wait_all();    // this warp's tiled stores are complete
  __syncwarp();
  pdl_trigger();                           // the next kernel may launch while this one drains
  settle_after_timeout(g.status, false);   // after a timeout, copies and MMAs may still be in flight
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, C::TMEM_COLS);
}

}  // namespace tc
}  // namespace evo

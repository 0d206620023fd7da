// Device code of the cached denoiser.
//
// One persistent kernel runs whole action queries.  A "job" is a group of g
// samples that share one schedule; a thread-block cluster of C CTAs runs the
// job's complete T-step reverse-diffusion loop (Sec. 3.1: T steps, B = 3L
// cacheable units) without returning to the host:
//
//   for t in 0..T-1:
//     a = x W_in + b_in + P_pos                      (this CTA's E/C columns)
//     for b in 0..3L-1:                              (Eq. 1)
//       (b,t) in S ? r = branch_b(a), c_b <- r, a += r
//                  : a += c_b                        (skip: a local add)
//     eps = LN_f(a) W_head + b_head ; x <- sampler step(x, eps, z_t)
//
// The residual stream a is distributed over the cluster by columns: each CTA
// owns E/C columns of a and of every unit's cache c_b (in shared memory when
// the slice fits, else in global memory), so a skipped cell is a local add.
// A refreshed unit needs two cluster exchanges, both done with bulk
// asynchronous copies from this CTA's shared memory into the other CTAs'
// (cp.async.bulk shared::cta -> shared::cluster, one per destination) that
// count their bytes on the receiver's mbarrier -- no fences and no
// cluster-wide barriers:
//   1. all-gather of a, so every CTA normalises full rows (LayerNorm);
//   2. reduce-scatter of the second matmul's partial sums, so every CTA
//      finishes its own columns of r = branch output.
// In between each CTA computes its share of the branch: attention -- the
// queries/keys of its head and its slice of head dimensions; FFN -- its slice
// of the hidden layer.  The order of the exchanges makes every buffer's reuse
// safe: a CTA can only send into a buffer again after it has received data
// that the receiver sends once it has finished reading that buffer.
//
// Weights never pass through registers on their way in: a producer warp per
// CTA walks the same schedule and streams, for every refreshed unit only, the
// CTA's pre-packed weight slices (with the unit's LayerNorm gain/shift and
// biases in front) through a ring of shared-memory slots with bulk
// asynchronous copies (cp.async.bulk + mbarrier transaction counts).  Skipped
// units generate no weight traffic, so time follows the schedule.
//
// bf16 mode: GEMM operands bf16, mma.sync m16n8k16 with fp32 accumulation
// (rows per job are 16..32, far below a tcgen05 tile; the cost here is weight
// streaming and on-chip latency, not tensor throughput).  fp32 mode: FFMA.
// Caches are stored in the GEMM operand type.

#include "evo_internal.h"

namespace evo {

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t addr, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(addr), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_try_wait_acq_cluster(uint32_t addr, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(addr), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ uint32_t mapa(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

__device__ __forceinline__ void mbar_arrive_cluster(uint32_t remote_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote_addr) : "memory");
}

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// asynchronous store into (possibly remote) shared memory; the bytes are
// counted on the mbarrier `rbar` of the receiving CTA
__device__ __forceinline__ void st_async_v4(uint32_t raddr, float4 v, uint32_t rbar) {
  asm volatile(
      "st.async.weak.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
          raddr),
      "r"(__float_as_uint(v.x)), "r"(__float_as_uint(v.y)), "r"(__float_as_uint(v.z)), "r"(__float_as_uint(v.w)),
      "r"(rbar)
      : "memory");
}

__device__ __forceinline__ void st_async_v2(uint32_t raddr, float a, float b, uint32_t rbar) {
  asm volatile("st.async.weak.shared::cluster.mbarrier::complete_tx::bytes.v2.b32 [%0], {%1, %2}, [%3];" ::"r"(
                   raddr),
               "r"(__float_as_uint(a)), "r"(__float_as_uint(b)), "r"(rbar)
               : "memory");
}

__device__ __forceinline__ void st_async_f32(uint32_t raddr, float a, uint32_t rbar) {
  asm volatile("st.async.weak.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];" ::"r"(raddr),
               "r"(__float_as_uint(a)), "r"(rbar)
               : "memory");
}

// bulk copy of `bytes` from this CTA's shared memory to a cluster-mapped
// address; completion counted on the (cluster-mapped) mbarrier of the receiver
__device__ __forceinline__ void bulk_s2c(uint32_t dst, const void* src, uint32_t bytes, uint32_t rbar) {
  asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "r"(smem_u32(src)), "r"(bytes), "r"(rbar)
               : "memory");
}

// orders this thread's generic-proxy shared-memory writes before later bulk copies
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ void fence_cluster() { asm volatile("fence.acq_rel.cluster;" ::: "memory"); }

__device__ __forceinline__ void bar_compute() { asm volatile("bar.sync 1, %0;" ::"n"(NCT) : "memory"); }

__device__ __forceinline__ void hw_cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint32_t cluster_idx() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint32_t cluster_count() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}

__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint2 b) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b.x), "r"(b.y));
}

// reductions over groups of G consecutive lanes (G a power of two <= 32)
template <int G>
__device__ __forceinline__ float group_sum(float v) {
#pragma unroll
  for (int o = G / 2; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float group_sum_dyn(float v, int G) {
  for (int o = G / 2; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float group_max_dyn(float v, int G) {
  for (int o = G / 2; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

__device__ __forceinline__ float gelu_erf(float x) { return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f)); }

__device__ __forceinline__ float mish(float x) {
  const float sp = x > 20.0f ? x : log1pf(expf(x));
  return x * tanhf(sp);
}

// A bounded wait: after ~2 s of SM cycles the wait gives up, records
// ST_TIMEOUT and lets the thread continue so that every CTA still reaches the
// same synchronisation points and the kernel ends.
constexpr long long WAIT_LIMIT = 4000000000LL;

struct Ctx {
  uint8_t* smem;
  uint64_t* full;
  uint64_t* empty;
  uint64_t* cbar;
  uint64_t* xg;    // receives the all-gather of a for a unit (and the head when it uses ablk)
  uint64_t* xr;    // receives the reduce-scatter partial sums
  uint64_t* xh;    // receives the head's all-gather, two barriers by step parity
  uint32_t q;      // slab counter (same sequence as the producer)
  uint32_t cph, pg, pr, ph0, ph1;   // phase parities
  int dead;
  int c, tid, warp, lane;
  // this thread's 16-byte chunk of a memory key/value staging (kv_i < 0: none):
  // sample kv_i of the job, token kv_tok, float offset kv_src within the token's
  // [k | v] row, float offset kv_dst within the staging slot; kv_base = the
  // token's rows for the current job (timestep table or observation keys/values)
  int kv_i, kv_tok, kv_src, kv_dst;
  const float* kv_base;
};

__device__ __forceinline__ void wait_parity(uint32_t addr, uint32_t parity, bool cluster_acq, Ctx& cx,
                                            int* status) {
  if (cx.dead) return;
  if (cluster_acq ? mbar_try_wait_acq_cluster(addr, parity) : mbar_try_wait(addr, parity)) return;
  const long long t0 = clock64();
  while (!(cluster_acq ? mbar_try_wait_acq_cluster(addr, parity) : mbar_try_wait(addr, parity))) {
    if (clock64() - t0 > WAIT_LIMIT) {
      atomicOr(status, ST_TIMEOUT);
      cx.dead = 1;
      return;
    }
  }
}

// cluster-wide barrier among the compute warps only (the producer warp runs
// ahead); used where no data exchange orders a buffer's reuse
__device__ __forceinline__ void csync(const JobParams& p, Ctx& cx) {
  fence_cluster();
  bar_compute();
  if (cx.tid < p.C) mbar_arrive_cluster(mapa(smem_u32(cx.cbar), cx.tid));
  wait_parity(smem_u32(cx.cbar), cx.cph, true, cx, p.status);
  cx.cph ^= 1u;
}

// receive one exchange phase of `bytes` on barrier `bar`
__device__ __forceinline__ void exchange_wait(const JobParams& p, Ctx& cx, uint64_t* bar, uint32_t& parity,
                                              uint32_t bytes) {
  if (cx.tid == 0) mbar_arrive_expect_tx(bar, bytes);
  wait_parity(smem_u32(bar), parity, true, cx, p.status);
  parity ^= 1u;
}

__device__ __forceinline__ const uint8_t* ring_acquire(const JobParams& p, Ctx& cx) {
  const uint32_t slot = cx.q % p.nslot;
  const uint32_t ph = (cx.q / p.nslot) & 1u;
  wait_parity(smem_u32(&cx.full[slot]), ph, false, cx, p.status);
  return cx.smem + p.sm.ring + slot * p.slot_bytes;
}

__device__ __forceinline__ void ring_release(const JobParams& p, Ctx& cx) {
  __syncwarp();
  if (cx.lane == 0) mbar_arrive(&cx.empty[cx.q % p.nslot]);
  cx.q++;
}

// slab s of a piece: first k-tile, k-tile count, byte offset and bytes (no divisions)
__device__ __forceinline__ SlabInfo slab_of(const PieceInfo& pi, int s) {
  if (s == 0) return SlabInfo{0, pi.k0, 0, pi.hdr + pi.k0 * pi.ktb};
  const int kt0 = pi.k0 + (s - 1) * pi.kps;
  const int n = min(pi.kps, pi.K / 16 - kt0);
  return SlabInfo{kt0, n, pi.hdr + kt0 * pi.ktb, n * pi.ktb};
}

// ---------------------------------------------------------------------------
// producer: stream the weight slabs of refreshed units, in schedule order
// ---------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ void producer(const JobParams& p, Ctx& cx, uint32_t cid, uint32_t ncl) {
  uint32_t q = 0;
  for (int job = cid; job < p.n_jobs; job += ncl) {
    const int s0 = min(job * p.g, p.samples - 1);
    const uint8_t* S = p.S + (long long)(s0 / p.per_sched) * p.S_stride;
    uint64_t valid = 0;
    for (int t = 0; t < p.T; ++t) {
      for (int b = 0; b < p.U; ++b) {
        const int row = (p.S_rows == p.U) ? b : b / 3;
        const bool vb = (valid >> b) & 1ull;
        if (!(S[row * p.T + t] != 0 || (p.force && !vb))) continue;   // same rule as the compute warps
        valid |= 1ull << b;
        const int l = b / 3, u = b % 3;
        for (int piece = 0; piece < 2; ++piece) {
          const PieceInfo& pi = p.pc[u][piece];
          const uint8_t* src = p.wpack + (long long)cx.c * p.cta_stride + (long long)l * p.layer_stride +
                               p.poff[u][piece];
          for (int s = 0; s < pi.ns; ++s) {
            const SlabInfo si = slab_of(pi, s);
            const uint32_t slot = q % p.nslot;
            const uint32_t ph = (q / p.nslot) & 1u;
            if (!mbar_try_wait(smem_u32(&cx.empty[slot]), ph ^ 1u)) {
              // the producer runs ahead of the compute warps: poll gently
              const long long t0 = clock64();
              while (!cx.dead && !mbar_try_wait(smem_u32(&cx.empty[slot]), ph ^ 1u)) {
                __nanosleep(64);
                if (clock64() - t0 > WAIT_LIMIT) {
                  atomicOr(p.status, ST_TIMEOUT);
                  cx.dead = 1;
                }
              }
            }
            mbar_arrive_expect_tx(&cx.full[slot], (uint32_t)si.bytes);
            bulk_g2s(cx.smem + p.sm.ring + slot * p.slot_bytes, src + si.off, (uint32_t)si.bytes, &cx.full[slot]);
            ++q;
          }
        }
      }
    }
  }
  // drain: every slab issued has landed before this CTA may exit (bounded waits)
  const uint32_t first = q > (uint32_t)p.nslot ? q - p.nslot : 0u;
  for (uint32_t k = first; k < q; ++k)
    wait_parity(smem_u32(&cx.full[k % p.nslot]), (k / p.nslot) & 1u, false, cx, p.status);
}

// ---------------------------------------------------------------------------
// GEMMs over streamed weight slabs.  A: shared memory, row-major.
// bf16: warp w owns n-tiles w, w+8, ...; NTW = n-tiles per warp (compile time).
// ---------------------------------------------------------------------------
template <int MT, int NTW>
__device__ __forceinline__ void gemm_bf16(const JobParams& p, Ctx& cx, const __nv_bfloat16* A, int lda,
                                          const PieceInfo& pi, const uint8_t* slab0, float (&acc)[MT][NTW][4]) {
  const int NT = pi.N >> 3;
#pragma unroll
  for (int m = 0; m < MT; ++m)
#pragma unroll
    for (int i = 0; i < NTW; ++i)
#pragma unroll
      for (int r = 0; r < 4; ++r) acc[m][i][r] = 0.f;
  const __nv_bfloat16* arow = A + (cx.lane & 15) * lda + (cx.lane >> 4) * 8;
  for (int s = 0; s < pi.ns; ++s) {
    const uint8_t* sl = s == 0 ? slab0 : ring_acquire(p, cx);
    const SlabInfo si = slab_of(pi, s);
    const uint8_t* wt = sl + (s == 0 ? pi.hdr : 0) + cx.lane * 8;
#pragma unroll 2
    for (int kk = 0; kk < si.nkt; ++kk) {
      const int kt = si.kt0 + kk;
      uint32_t a[MT][4];
#pragma unroll
      for (int m = 0; m < MT; ++m) ldmatrix_x4(a[m], arow + m * 16 * lda + kt * 16);
      uint2 bf[NTW];
#pragma unroll
      for (int i = 0; i < NTW; ++i) {
        const int nt = cx.warp + i * NCW;
        bf[i] = nt < NT ? *reinterpret_cast<const uint2*>(wt + (size_t)(kk * NT + nt) * 256) : make_uint2(0u, 0u);
      }
#pragma unroll
      for (int i = 0; i < NTW; ++i)
        if (cx.warp + i * NCW < NT) {
#pragma unroll
          for (int m = 0; m < MT; ++m) mma_bf16(acc[m][i], a[m], bf[i]);
        }
    }
    ring_release(p, cx);
  }
}

constexpr int F32_MAXO = 16;

__device__ __forceinline__ void gemm_f32(const JobParams& p, Ctx& cx, const float* A, int lda, const PieceInfo& pi,
                                         const uint8_t* slab0, float (&acc)[F32_MAXO]) {
  const int M = p.M, N = pi.N;
  int mi[F32_MAXO], ni[F32_MAXO];
  const int nout = M * N;
#pragma unroll
  for (int i = 0; i < F32_MAXO; ++i) {
    const int o = cx.tid + i * NCT;
    mi[i] = o < nout ? o / N : 0;
    ni[i] = o < nout ? o % N : 0;
    acc[i] = 0.f;
  }
  for (int s = 0; s < pi.ns; ++s) {
    const uint8_t* sl = s == 0 ? slab0 : ring_acquire(p, cx);
    const SlabInfo si = slab_of(pi, s);
    const float* W = reinterpret_cast<const float*>(sl + (s == 0 ? pi.hdr : 0));
    const int rows = si.nkt * 16;
    for (int r = 0; r < rows; ++r) {
      const int k = si.kt0 * 16 + r;
#pragma unroll
      for (int i = 0; i < F32_MAXO; ++i)
        if (cx.tid + i * NCT < nout) acc[i] = fmaf(A[mi[i] * lda + k], W[r * N + ni[i]], acc[i]);
    }
    ring_release(p, cx);
  }
}

// ---------------------------------------------------------------------------
// compute-warp building blocks
// ---------------------------------------------------------------------------

// Send one block of M*Ec floats to every CTA r of the cluster: block
// src + r*src_stride lands in CTA r at dst + c*blk (c = this CTA), counted on
// r's barrier `rbar`.  The writers of src have executed fence_proxy_async()
// and a bar_compute() before this call.
__device__ __forceinline__ void send_blocks(const JobParams& p, Ctx& cx, const float* src, int src_stride,
                                            const float* dst, uint64_t* rbar) {
  if (cx.tid < p.C) {
    const uint32_t r = (uint32_t)cx.tid;
    bulk_s2c(mapa(smem_u32(dst + cx.c * p.blk), r), src + r * src_stride, (uint32_t)(p.M * p.Ec * 4),
             mapa(smem_u32(rbar), r));
  }
}

// LayerNorm of rows m < M (half a warp per row).  Row m is read from the
// gathered blocks (column col of the row is in block col/Ec) and written to the
// A operand xln in type T.
template <typename T>
__device__ __forceinline__ void layernorm_rows(const JobParams& p, Ctx& cx, const float* blk, T* xln,
                                               const float* gam, const float* bet) {
  const int half = cx.lane >> 4, hl = cx.lane & 15;
  const int nv = p.E >> 6;                      // float4 chunks per lane
  for (int m0 = 0; m0 < p.M; m0 += 2 * NCW) {
    if (m0 + cx.warp * 2 >= p.M) break;           // warp-uniform (M is even)
    const int m = m0 + cx.warp * 2 + half;
    float4 v[8];
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j < nv) {
        const int col = 4 * (hl + 16 * j);
        v[j] = *reinterpret_cast<const float4*>(blk + (col >> p.lEc) * p.blk + (m << p.lEc) + (col & (p.Ec - 1)));
        s += (v[j].x + v[j].y) + (v[j].z + v[j].w);
      }
    const float mean = group_sum<16>(s) * p.invE;
    float s2 = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j < nv) {
        const float a = v[j].x - mean, b = v[j].y - mean, c = v[j].z - mean, d = v[j].w - mean;
        s2 += (a * a + b * b) + (c * c + d * d);
      }
    const float rstd = rsqrtf(group_sum<16>(s2) * p.invE + 1e-5f);
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j < nv) {
        const int col = 4 * (hl + 16 * j);
        const float4 g = *reinterpret_cast<const float4*>(gam + col);
        const float4 bb = *reinterpret_cast<const float4*>(bet + col);
        const float y0 = (v[j].x - mean) * rstd * g.x + bb.x, y1 = (v[j].y - mean) * rstd * g.y + bb.y;
        const float y2 = (v[j].z - mean) * rstd * g.z + bb.z, y3 = (v[j].w - mean) * rstd * g.w + bb.w;
        T* dst = xln + m * p.lda + col;
        if constexpr (sizeof(T) == 2) {
          __nv_bfloat162 lo = __floats2bfloat162_rn(y0, y1), hi = __floats2bfloat162_rn(y2, y3);
          uint2 pk;
          pk.x = *reinterpret_cast<uint32_t*>(&lo);
          pk.y = *reinterpret_cast<uint32_t*>(&hi);
          *reinterpret_cast<uint2*>(dst) = pk;
        } else {
          *reinterpret_cast<float4*>(dst) = make_float4(y0, y1, y2, y3);
        }
      }
  }
}

template <typename T>
struct Kern {
  static constexpr bool BF = sizeof(T) == 2;

  __device__ __forceinline__ static T* cache_ptr(const JobParams& p, Ctx& cx, int job, int b) {
    if (p.sm.cs >= 0) return reinterpret_cast<T*>(cx.smem + p.sm.cs) + (long long)b * p.M * p.Ec;
    return reinterpret_cast<T*>(p.cache) + ((long long)(job * p.U + b) * p.C + cx.c) * p.M * p.Ec;
  }

  // ---- first GEMM + epilogue ------------------------------------------------
  // A = xln.  SA / CA: f32 rows of q|k|v (SA) or q (CA) + bias; FFN:
  // T(gelu(. + bias)).  The output region aliases xln, so all warps finish
  // their k-loop before any epilogue writes.
  template <int MT, int NTW>
  __device__ __forceinline__ static void gemm1_t(const JobParams& p, Ctx& cx, int u, const uint8_t* slab0) {
    const T* xln = reinterpret_cast<const T*>(cx.smem + p.sm.xln);
    const int N = p.n1[u];
    const float* bias = reinterpret_cast<const float*>(slab0) + 2 * p.E;
    float* g1 = reinterpret_cast<float*>(cx.smem + p.sm.xln);
    T* hid = reinterpret_cast<T*>(cx.smem + p.sm.xln);
    const int NT = N >> 3;
    float2 bv[NTW];
#pragma unroll
    for (int i = 0; i < NTW; ++i) {
      const int nt = cx.warp + i * NCW;
      bv[i] = nt < NT ? *reinterpret_cast<const float2*>(bias + nt * 8 + 2 * (cx.lane & 3)) : make_float2(0.f, 0.f);
    }
    float acc[MT][NTW][4];
    gemm_bf16<MT, NTW>(p, cx, reinterpret_cast<const __nv_bfloat16*>(xln), p.lda, p.pc[u][0], slab0, acc);
    bar_compute();
#pragma unroll
    for (int i = 0; i < NTW; ++i) {
      const int nt = cx.warp + i * NCW;
      if (nt < NT) {
        const int n = nt * 8 + 2 * (cx.lane & 3);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int m = mt * 16 + (cx.lane >> 2) + 8 * h;
            if (m < p.M) {
              const float v0 = acc[mt][i][2 * h] + bv[i].x, v1 = acc[mt][i][2 * h + 1] + bv[i].y;
              if (u == 2) {
                *reinterpret_cast<__nv_bfloat162*>(hid + m * p.ldh + n) =
                    __floats2bfloat162_rn(gelu_erf(v0), gelu_erf(v1));
              } else {
                *reinterpret_cast<float2*>(g1 + m * p.ldg1 + n) = make_float2(v0, v1);
              }
            }
          }
      }
    }
  }

  template <int MT>
  __device__ __forceinline__ static void gemm1(const JobParams& p, Ctx& cx, int u, const uint8_t* slab0) {
    if constexpr (BF) {
      const int ntw = ((p.n1[u] >> 3) + NCW - 1) / NCW;
      if (ntw <= 1) gemm1_t<MT, 1>(p, cx, u, slab0);
      else if (ntw == 2) gemm1_t<MT, 2>(p, cx, u, slab0);
      else if (ntw == 3) gemm1_t<MT, 3>(p, cx, u, slab0);
      else if (MT == 1 || ntw == 4) gemm1_t<MT, 4>(p, cx, u, slab0);   // one 16-row tile: N <= 256 (host check)
      else gemm1_t<MT, 8>(p, cx, u, slab0);
    } else {
      const float* xln = reinterpret_cast<const float*>(cx.smem + p.sm.xln);
      const int N = p.n1[u];
      const float* bias = reinterpret_cast<const float*>(slab0) + 2 * p.E;
      float* g1 = reinterpret_cast<float*>(cx.smem + p.sm.xln);
      T* hid = reinterpret_cast<T*>(cx.smem + p.sm.xln);
      float bv[F32_MAXO];
#pragma unroll
      for (int i = 0; i < F32_MAXO; ++i) {
        const int o = cx.tid + i * NCT;
        bv[i] = o < p.M * N ? bias[o % N] : 0.f;
      }
      float acc[F32_MAXO];
      gemm_f32(p, cx, xln, p.lda, p.pc[u][0], slab0, acc);
      bar_compute();
#pragma unroll
      for (int i = 0; i < F32_MAXO; ++i) {
        const int o = cx.tid + i * NCT;
        if (o < p.M * N) {
          const int m = o / N, n = o % N;
          const float v = acc[i] + bv[i];
          if (u == 2)
            hid[m * p.ldh + n] = from_f<T>(gelu_erf(v));
          else
            g1[m * p.ldg1 + n] = v;
        }
      }
    }
  }

  // ---- second GEMM: partial sums over this CTA's K slice, staged in ablk
  // block layout (block r = columns r*Ec.. destined for CTA r)
  template <int MT, int NTW>
  __device__ __forceinline__ static void gemm2_t(const JobParams& p, Ctx& cx, int u) {
    const T* A = reinterpret_cast<const T*>(cx.smem + (u == 2 ? p.sm.xln : p.sm.oc));
    const int lda = u == 2 ? p.ldh : p.ldo;
    float* stage = reinterpret_cast<float*>(cx.smem + p.sm.ablk);
    float acc[MT][NTW][4];
    gemm_bf16<MT, NTW>(p, cx, reinterpret_cast<const __nv_bfloat16*>(A), lda, p.pc[u][1], ring_acquire(p, cx), acc);
    const int NT = p.E >> 3;
#pragma unroll
    for (int i = 0; i < NTW; ++i) {
      const int nt = cx.warp + i * NCW;
      if (nt < NT) {
        const int n = nt * 8 + 2 * (cx.lane & 3);
        float* dst = stage + (n >> p.lEc) * p.blk + (n & (p.Ec - 1));
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int m = mt * 16 + (cx.lane >> 2) + 8 * h;
            if (m < p.M)
              *reinterpret_cast<float2*>(dst + (m << p.lEc)) = make_float2(acc[mt][i][2 * h], acc[mt][i][2 * h + 1]);
          }
      }
    }
  }

  template <int MT>
  __device__ __forceinline__ static void gemm2(const JobParams& p, Ctx& cx, int u) {
    if constexpr (BF) {
      const int ntw = ((p.E >> 3) + NCW - 1) / NCW;
      if (ntw <= 1) gemm2_t<MT, 1>(p, cx, u);
      else if (ntw == 2) gemm2_t<MT, 2>(p, cx, u);
      else if (MT == 1 || ntw <= 4) gemm2_t<MT, 4>(p, cx, u);          // one 16-row tile: N <= 256 (host check)
      else gemm2_t<MT, 8>(p, cx, u);
    } else {
      const T* A = reinterpret_cast<const T*>(cx.smem + (u == 2 ? p.sm.xln : p.sm.oc));
      const int lda = u == 2 ? p.ldh : p.ldo;
      float* stage = reinterpret_cast<float*>(cx.smem + p.sm.ablk);
      float acc[F32_MAXO];
      gemm_f32(p, cx, reinterpret_cast<const float*>(A), lda, p.pc[u][1], ring_acquire(p, cx), acc);
#pragma unroll
      for (int i = 0; i < F32_MAXO; ++i) {
        const int o = cx.tid + i * NCT;
        if (o < p.M * p.E) {
          const int m = o / p.E, n = o % p.E;
          stage[(n >> p.lEc) * p.blk + (m << p.lEc) + (n & (p.Ec - 1))] = acc[i];
        }
      }
    }
  }

  // ---- attention for this CTA's head-dimension slice ------------------------
  // scores: one (query row, key) pair per thread, softmax over groups of G
  // lanes, probabilities to pb; then one output (row, dim) per thread.
  // SA: causal over the H tokens of the same sample (q, k of the CTA's head and
  // v of its slice, rows of the first GEMM's output).  CA: the 1 + n_obs memory
  // tokens in kvs.
  __device__ __forceinline__ static void attention(const JobParams& p, Ctx& cx, int u, const float* kvs) {
    const float* g1 = reinterpret_cast<const float*>(cx.smem + p.sm.xln);
    float* pb = reinterpret_cast<float*>(cx.smem + p.sm.pb);
    T* oc = reinterpret_cast<T*>(cx.smem + p.sm.oc);
    const float scale = 1.0f / sqrtf((float)p.dh);
    const int nk = u == 0 ? p.H : p.Cm;
    int lG = 0;
    while ((1 << lG) < nk) ++lG;
    const int G = 1 << lG;
    const int rows_per_pass = NCT >> lG;
    const int nd4 = p.dh >> 2;
    for (int base = 0; base < p.M; base += rows_per_pass) {
      const int m = base + (cx.tid >> lG), j = cx.tid & (G - 1);
      float s = -INFINITY;
      const bool live = m < p.M && j < nk;
      if (live) {
        const int i = m >> p.lH, qi = m & (p.H - 1);
        if (u != 0 || j <= qi) {
          const float4* q4 = reinterpret_cast<const float4*>(g1 + m * p.ldg1);
          const float4* k4 = u == 0 ? reinterpret_cast<const float4*>(g1 + ((i << p.lH) + j) * p.ldg1 + p.dh)
                                    : reinterpret_cast<const float4*>(kvs + (i * p.Cm + j) * p.kvw);
          float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
#pragma unroll 4
          for (int e = 0; e < nd4; ++e) {
            const float4 a = q4[e], b = k4[e];
            d0 = fmaf(a.x, b.x, d0);
            d1 = fmaf(a.y, b.y, d1);
            d2 = fmaf(a.z, b.z, d2);
            d3 = fmaf(a.w, b.w, d3);
          }
          s = ((d0 + d1) + (d2 + d3)) * scale;
        }
      }
      const float mx = group_max_dyn(s, G);
      const float ex = s == -INFINITY ? 0.f : expf(s - mx);
      const float sum = group_sum_dyn(ex, G);
      if (live) pb[m * PLD + j] = ex * __frcp_rn(sum);
    }
    bar_compute();
    for (int o = cx.tid; o < p.M * p.Ec; o += NCT) {
      const int m = o >> p.lEc, e = o & (p.Ec - 1);
      const int i = m >> p.lH, qi = m & (p.H - 1);
      const int nj = u == 0 ? qi + 1 : p.Cm;
      const float* prow = pb + m * PLD;
      float a0 = 0.f, a1 = 0.f;
      int j = 0;
      if (u == 0) {
        const float* v = g1 + (i << p.lH) * p.ldg1 + 2 * p.dh + e;
        for (; j + 1 < nj; j += 2) {
          a0 = fmaf(prow[j], v[j * p.ldg1], a0);
          a1 = fmaf(prow[j + 1], v[(j + 1) * p.ldg1], a1);
        }
        if (j < nj) a0 = fmaf(prow[j], v[j * p.ldg1], a0);
      } else {
        const float* v = kvs + (i * p.Cm) * p.kvw + p.dh + e;
        for (; j < nj; ++j) a0 = fmaf(prow[j], v[j * p.kvw], a0);
      }
      oc[m * p.ldo + e] = from_f<T>(a0 + a1);
    }
  }

  // stage the memory tokens' keys (this CTA's head) and values (its slice) of
  // layer l at step t into kvs (cp.async; waited before use)
  __device__ __forceinline__ static void stage_kv(const JobParams& p, Ctx& cx, int l, int t, float* kvs) {
    if (cx.kv_i >= 0) {
      const float* src = cx.kv_base + (cx.kv_tok == 0 ? (long long)t * p.L * 2 * p.E : 0ll) + l * 2 * p.E + cx.kv_src;
      cp_async16(kvs + cx.kv_dst, src);
    }
  }

  // per-job part of the staging map (which sample's observation rows this thread copies)
  __device__ __forceinline__ static void stage_kv_job(const JobParams& p, Ctx& cx, int sample0) {
    if (cx.kv_i < 0) return;
    const int s = min(sample0 + cx.kv_i, p.samples - 1);
    cx.kv_base = cx.kv_tok == 0 ? p.kv_time
                                : p.kv_obs + ((long long)(s % p.obs_mod) * p.n_obs + (cx.kv_tok - 1)) * p.L * 2 * p.E;
  }

  // ---- one refreshed unit (Eq. 1, (b,t) in S) --------------------------------
  template <int MT>
  __device__ __forceinline__ static void unit(const JobParams& p, Ctx& cx, int job, int b, int t, int sample0) {
    const int l = b / 3, u = b % 3;
    float* ac = reinterpret_cast<float*>(cx.smem + p.sm.ac);
    float* ablk = reinterpret_cast<float*>(cx.smem + p.sm.ablk);
    float* kvs = reinterpret_cast<float*>(cx.smem + p.sm.kvs);
    if (u == 1) {
      if (p.kv_slots == 1) stage_kv(p, cx, l, t, kvs);
      else kvs += l * p.g * p.Cm * p.kvw;
    }
    // exchange 1: every CTA receives every CTA's columns of a
    fence_proxy_async();
    bar_compute();                     // ac final for this unit
    send_blocks(p, cx, ac, 0, ablk, cx.xg);
    exchange_wait(p, cx, cx.xg, cx.pg, (uint32_t)(p.M * p.E * 4));
    // slab 0 of piece 1: [gamma | beta | first bias | second-GEMM bias slice | k-tiles]
    const uint8_t* s1 = ring_acquire(p, cx);
    const float* hdr = reinterpret_cast<const float*>(s1);
    float b2[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int e = cx.tid + k * NCT;
      b2[k] = e < p.M * p.Ec ? hdr[2 * p.E + p.n1[u] + (e & (p.Ec - 1))] : 0.f;
    }
    layernorm_rows<T>(p, cx, ablk, reinterpret_cast<T*>(cx.smem + p.sm.xln), hdr, hdr + p.E);
    bar_compute();
    gemm1<MT>(p, cx, u, s1);
    if (u == 1) cp_async_wait_all();
    bar_compute();
    if (u != 2) {
      attention(p, cx, u, kvs);
      bar_compute();
    }
    gemm2<MT>(p, cx, u);
    // exchange 2: block r of the staged partial sums goes to CTA r
    fence_proxy_async();
    bar_compute();
    send_blocks(p, cx, ablk, p.blk, reinterpret_cast<const float*>(cx.smem + p.sm.rs), cx.xr);
    exchange_wait(p, cx, cx.xr, cx.pr, (uint32_t)(p.M * p.E * 4));
    // finish this CTA's columns: r = sum of partials + bias; c_b <- r; a += r
    const float* rs = reinterpret_cast<const float*>(cx.smem + p.sm.rs);
    T* cache = cache_ptr(p, cx, job, b);
    const int MEc = p.M * p.Ec;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int e = cx.tid + k * NCT;
      if (e < MEc) {
        float part[MAX_CLUSTER];
#pragma unroll
        for (int cc = 0; cc < MAX_CLUSTER; ++cc) part[cc] = cc < p.C ? rs[cc * p.blk + e] : 0.f;
#pragma unroll
        for (int w = MAX_CLUSTER / 2; w > 0; w >>= 1)
#pragma unroll
          for (int cc = 0; cc < w; ++cc) part[cc] += part[cc + w];
        const float r = part[0] + b2[k];
        cache[e] = from_f<T>(r);
        ac[e] += r;
        if (p.trace) {
          const int m = e >> p.lEc, j = e & (p.Ec - 1);
          const int s = sample0 + (m >> p.lH);
          if (s < p.samples)
            p.trace[(((long long)t * p.U + b) * p.samples + s) * p.H * p.E + (m & (p.H - 1)) * p.E + cx.c * p.Ec + j] = r;
        }
      }
    }
  }

  // ---- skipped units b0..b1-1: a += c_b on this CTA's columns (in unit order) ---
  __device__ __forceinline__ static void skip_run(const JobParams& p, Ctx& cx, int job, int b0, int b1, int t,
                                                  int sample0, uint64_t valid) {
    float* ac = reinterpret_cast<float*>(cx.smem + p.sm.ac);
    const int MEc = p.M * p.Ec;
    // units of the run whose cache holds a value (bit k = unit b0 + k)
    const uint32_t live = (uint32_t)((valid >> b0) & ((1ull << (b1 - b0)) - 1ull));
    const T* cb = cache_ptr(p, cx, job, b0);
    const long long cstride = p.sm.cs >= 0 ? (long long)MEc : (long long)p.C * MEc;
    for (int e = cx.tid; e < MEc; e += NCT) {
      float cv[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) cv[k] = ((live >> k) & 1u) ? to_f<T>(cb[k * cstride + e]) : 0.f;
      float a = ac[e];
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if ((live >> k) & 1u) a += cv[k];
      ac[e] = a;
      if (p.trace) {
        const int m = e >> p.lEc, j = e & (p.Ec - 1);
        const int s = sample0 + (m >> p.lH);
        if (s < p.samples) {
#pragma unroll
          for (int k = 0; k < 8; ++k)
            if (b0 + k < b1)
              p.trace[(((long long)t * p.U + b0 + k) * p.samples + s) * p.H * p.E + (m & (p.H - 1)) * p.E +
                      cx.c * p.Ec + j] = cv[k];
        }
      }
    }
  }

  // ---- output head + sampler step ---------------------------------------------
  __device__ __forceinline__ static void head_step(const JobParams& p, Ctx& cx, int t, const float4 tab0,
                                                   const float4 tab1) {
    float* ac = reinterpret_cast<float*>(cx.smem + p.sm.ac);
    float* x = reinterpret_cast<float*>(cx.smem + p.sm.x);
    const float* z = reinterpret_cast<const float*>(cx.smem + p.sm.z);
    const float* cst = reinterpret_cast<const float*>(cx.smem + p.sm.cst);
    const float* lnf_g = cst + p.A * p.Ec + p.Ec + p.H * p.Ec;
    const float* lnf_b = lnf_g + p.E;
    const float* head_b = lnf_b + p.E;
    const float* hw = p.headw_smem ? head_b + ((p.A + 3) & ~3) : p.vec + p.v_headw;
    const float* hb;
    if (p.head_sep) {
      // double-buffered by step parity: source, landing blocks and barrier
      const int par = t & 1;
      float* src = reinterpret_cast<float*>(cx.smem + p.sm.hsrc) + par * p.M * p.Ec;
      for (int e = cx.tid; e < p.M * p.Ec; e += NCT) src[e] = ac[e];
      hb = reinterpret_cast<const float*>(cx.smem + p.sm.hblk) + par * p.C * p.blk;
      fence_proxy_async();
      bar_compute();
      send_blocks(p, cx, src, 0, hb, cx.xh + par);
      exchange_wait(p, cx, cx.xh + par, par ? cx.ph1 : cx.ph0, (uint32_t)(p.M * p.E * 4));
    } else {
      hb = reinterpret_cast<const float*>(cx.smem + p.sm.ablk);
      fence_proxy_async();
      bar_compute();
      send_blocks(p, cx, ac, 0, hb, cx.xg);
      exchange_wait(p, cx, cx.xg, cx.pg, (uint32_t)(p.M * p.E * 4));
    }
    cp_async_wait_all();
    bar_compute();
    const float inv_sa = tab0.x, s1 = tab0.y, cx0 = tab0.z, cxt = tab0.w, sig = tab1.x;
    const float sab = tab1.y, sabp = tab1.z, s1p = tab1.w;
    const int half = cx.lane >> 4, hl = cx.lane & 15;
    const int nv = p.E >> 6;
    for (int m0 = 0; m0 < p.M; m0 += 2 * NCW) {
      if (m0 + cx.warp * 2 >= p.M) break;
      const int m = m0 + cx.warp * 2 + half;
      float4 v[8];
      float s = 0.f;
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (j < nv) {
          const int col = 4 * (hl + 16 * j);
          v[j] = *reinterpret_cast<const float4*>(hb + (col >> p.lEc) * p.blk + (m << p.lEc) + (col & (p.Ec - 1)));
          s += (v[j].x + v[j].y) + (v[j].z + v[j].w);
        }
      const float mean = group_sum<16>(s) * p.invE;
      float s2 = 0.f;
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (j < nv) {
          const float a = v[j].x - mean, b = v[j].y - mean, c = v[j].z - mean, d = v[j].w - mean;
          s2 += (a * a + b * b) + (c * c + d * d);
        }
      const float rstd = rsqrtf(group_sum<16>(s2) * p.invE + 1e-5f);
      // normalised values of this lane's columns, then one reduced dot per action dim
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (j < nv) {
          const int col = 4 * (hl + 16 * j);
          v[j].x = (v[j].x - mean) * rstd * lnf_g[col] + lnf_b[col];
          v[j].y = (v[j].y - mean) * rstd * lnf_g[col + 1] + lnf_b[col + 1];
          v[j].z = (v[j].z - mean) * rstd * lnf_g[col + 2] + lnf_b[col + 2];
          v[j].w = (v[j].w - mean) * rstd * lnf_g[col + 3] + lnf_b[col + 3];
        }
      float eps = 0.f;
      for (int a = 0; a < p.A; ++a) {
        float part = 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j)
          if (j < nv) {
            const float* w = hw + 4 * (hl + 16 * j) * p.A + a;
            part = fmaf(v[j].x, w[0], part);
            part = fmaf(v[j].y, w[p.A], part);
            part = fmaf(v[j].z, w[2 * p.A], part);
            part = fmaf(v[j].w, w[3 * p.A], part);
          }
        const float e = group_sum<16>(part);
        if (hl == a) eps = e + head_b[a];
      }
      if (hl < p.A) {
        const float xv = x[m * p.A + hl];
        float x0 = (xv - s1 * eps) * inv_sa;
        x0 = fminf(1.0f, fmaxf(-1.0f, x0));
        float xn;
        if (p.sampler == 0) {
          xn = cx0 * x0 + cxt * xv + sig * z[m * p.A + hl];
        } else {
          xn = sabp * x0 + s1p * ((xv - sab * x0) / s1);
        }
        x[m * p.A + hl] = xn;
      }
    }
    if (!p.head_sep) csync(p, cx);                    // ablk is the next gather's landing zone
    bar_compute();
  }

  template <int MT>
  __device__ __forceinline__ static void compute(const JobParams& p, Ctx& cx, uint32_t cid, uint32_t ncl) {
    float* ac = reinterpret_cast<float*>(cx.smem + p.sm.ac);
    float* x = reinterpret_cast<float*>(cx.smem + p.sm.x);
    float* z = reinterpret_cast<float*>(cx.smem + p.sm.z);
    uint64_t* sch = reinterpret_cast<uint64_t*>(cx.smem + p.sm.sch);
    float* kvs = reinterpret_cast<float*>(cx.smem + p.sm.kvs);
    const float* cst = reinterpret_cast<const float*>(cx.smem + p.sm.cst);
    const float* c_inw = cst;
    const float* c_inb = cst + p.A * p.Ec;
    const float* c_pos = c_inb + p.Ec;
    for (int job = cid; job < p.n_jobs; job += ncl) {
      const int sample0 = job * p.g;
      const int s_first = min(sample0, p.samples - 1);
      const uint8_t* S = p.S + (long long)(s_first / p.per_sched) * p.S_stride;
      // the job's lattice as one refresh mask per step, and the initial x
      for (int t = cx.tid; t < p.T; t += NCT) {
        uint64_t mask = 0;
        for (int b = 0; b < p.U; ++b) {
          const int row = (p.S_rows == p.U) ? b : b / 3;
          if (S[row * p.T + t] != 0) mask |= 1ull << b;
        }
        sch[t] = mask;
      }
      for (int v = cx.tid; v < p.M * p.A; v += NCT) {
        const int m = v / p.A;
        const int s = min(sample0 + (m >> p.lH), p.samples - 1);
        x[v] = p.noise[((long long)(s % p.obs_mod) * p.H + (m & (p.H - 1))) * p.A + (v % p.A)];
      }
      stage_kv_job(p, cx, sample0);
      bar_compute();
      uint64_t valid = 0;
      for (int t = 0; t < p.T; ++t) {
        const uint64_t st = sch[t];
        const uint64_t refresh = st | (p.force ? ~valid : 0ull);
        // sampler coefficients of this step (used at the head)
        const float4 tab0 = *reinterpret_cast<const float4*>(p.stab + t * 8);
        const float4 tab1 = *reinterpret_cast<const float4*>(p.stab + t * 8 + 4);
        // stage z_t (DDPM) and, when every layer has a slot, the memory keys/values
        // of this step's refreshed cross-attention units
        if (p.sampler == 0) {
          const int per = p.H * p.A / 4;
          for (int v = cx.tid; v < p.g * per; v += NCT) {
            const int i = v / per, w = v - i * per;
            const int s = min(sample0 + i, p.samples - 1);
            cp_async16(z + i * p.H * p.A + 4 * w,
                       p.noise + ((long long)(1 + t) * p.obs_mod + (s % p.obs_mod)) * p.H * p.A + 4 * w);
          }
        }
        if (p.kv_slots > 1)
          for (int l = 0; l < p.L; ++l)
            if ((refresh >> (3 * l + 1)) & 1ull) stage_kv(p, cx, l, t, kvs + l * p.g * p.Cm * p.kvw);
        // input embedding into this CTA's columns
        for (int e = cx.tid; e < p.M * p.Ec; e += NCT) {
          const int m = e >> p.lEc, j = e & (p.Ec - 1);
          float acc = 0.f;
          for (int a = 0; a < p.A; ++a) acc = fmaf(x[m * p.A + a], c_inw[a * p.Ec + j], acc);
          ac[e] = acc + c_inb[j] + c_pos[(m & (p.H - 1)) * p.Ec + j];
        }
        int b = 0;
        while (b < p.U) {
          if ((refresh >> b) & 1ull) {
            valid |= 1ull << b;
            unit<MT>(p, cx, job, b, t, sample0);
            ++b;
          } else {
            int b1 = b + 1;
            while (b1 < p.U && b1 - b < 8 && !((refresh >> b1) & 1ull)) ++b1;
            skip_run(p, cx, job, b, b1, t, sample0, valid);
            b = b1;
          }
        }
        head_step(p, cx, t, tab0, tab1);
      }
      // write the finished chunk
      if (cx.c == 0) {
        for (int v = cx.tid; v < p.M * p.A; v += NCT) {
          const int s = sample0 + v / (p.H * p.A);
          if (s < p.samples) p.out[(long long)sample0 * p.H * p.A + v] = x[v];
        }
      }
      bar_compute();
    }
  }
};

// MT = 16-row tiles per job (1: up to 16 rows, 2: up to 32): one instantiation
// per tile count keeps each launch's code and register budget to its own shapes
template <typename T, int MT>
__global__ void __launch_bounds__(NTHREADS, 1) job_kernel(const __grid_constant__ JobParams p) {
  extern __shared__ __align__(128) uint8_t smem[];
  Ctx cx;
  cx.smem = smem;
  cx.tid = threadIdx.x;
  cx.warp = threadIdx.x >> 5;
  cx.lane = threadIdx.x & 31;
  cx.c = (int)cluster_ctarank();
  cx.full = reinterpret_cast<uint64_t*>(smem + p.sm.bars);
  cx.empty = cx.full + p.nslot;
  cx.cbar = cx.full + 2 * p.nslot;
  cx.xg = cx.cbar + 1;
  cx.xr = cx.cbar + 2;
  cx.xh = cx.cbar + 3;
  cx.q = 0;
  cx.cph = cx.pg = cx.pr = cx.ph0 = cx.ph1 = 0;
  cx.dead = 0;
  {
    // staging map: chunk v = tid over [g][1+n_obs][k chunks (dh/4) | v chunks (Ec/4)]
    const int kq = p.dh >> 2, per_tok = kq + (p.Ec >> 2);
    const int v = threadIdx.x;
    cx.kv_i = -1;
    cx.kv_base = nullptr;
    if (v < p.g * p.Cm * per_tok) {
      const int i = v / (p.Cm * per_tok);
      const int rem = v - i * p.Cm * per_tok;
      const int tok = rem / per_tok, w = rem - tok * per_tok;
      const int head = (cx.c * p.Ec) / p.dh;
      cx.kv_i = i;
      cx.kv_tok = tok;
      cx.kv_src = w < kq ? head * p.dh + 4 * w : p.E + cx.c * p.Ec + 4 * (w - kq);
      cx.kv_dst = (i * p.Cm + tok) * p.kvw + (w < kq ? 4 * w : p.dh + 4 * (w - kq));
    }
  }
  const uint32_t cid = cluster_idx(), ncl = cluster_count();

  if (threadIdx.x == 0) {
    for (int i = 0; i < p.nslot; ++i) {
      mbar_init(&cx.full[i], 1);
      mbar_init(&cx.empty[i], NCW);
    }
    mbar_init(cx.cbar, p.C);
    mbar_init(cx.xg, 1);
    mbar_init(cx.xr, 1);
    mbar_init(cx.xh, 1);
    mbar_init(cx.xh + 1, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // zero the operand and exchange buffers once: padded rows and columns must read as 0
  for (int v = threadIdx.x; v < (p.sm.ac - p.sm.ablk) / 16; v += NTHREADS)
    reinterpret_cast<float4*>(smem + p.sm.ablk)[v] = make_float4(0.f, 0.f, 0.f, 0.f);
  // per-kernel constants: in_w[:, cols], in_b[cols], pos[:, cols], lnf_g, lnf_b, head_b, head_w
  {
    float* cst = reinterpret_cast<float*>(smem + p.sm.cst);
    const int c0 = cx.c * p.Ec;
    for (int v = threadIdx.x; v < p.A * p.Ec; v += NTHREADS)
      cst[v] = p.vec[p.v_inw + (v / p.Ec) * p.E + c0 + (v % p.Ec)];
    float* d = cst + p.A * p.Ec;
    for (int v = threadIdx.x; v < p.Ec; v += NTHREADS) d[v] = p.vec[p.v_inb + c0 + v];
    d += p.Ec;
    for (int v = threadIdx.x; v < p.H * p.Ec; v += NTHREADS) d[v] = p.vec[p.v_pos + (v / p.Ec) * p.E + c0 + (v % p.Ec)];
    d += p.H * p.Ec;
    for (int v = threadIdx.x; v < p.E; v += NTHREADS) {
      d[v] = p.vec[p.v_lnfg + v];
      d[p.E + v] = p.vec[p.v_lnfb + v];
    }
    d += 2 * p.E;
    for (int v = threadIdx.x; v < p.A; v += NTHREADS) d[v] = p.vec[p.v_headb + v];
    d += (p.A + 3) & ~3;
    if (p.headw_smem)
      for (int v = threadIdx.x; v < p.E * p.A; v += NTHREADS) d[v] = p.vec[p.v_headw + v];
  }
  __syncthreads();
  hw_cluster_sync();
  const bool bad = p.sched_err != nullptr && *p.sched_err != 0;
  if (!bad) {
    if (cx.warp == NCW) {
      if (cx.lane == 0) producer<T>(p, cx, cid, ncl);
      __syncwarp();
    } else {
      Kern<T>::template compute<MT>(p, cx, cid, ncl);
    }
  }
  __syncwarp();
  hw_cluster_sync();
}

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
  if (p.head_sep) {
    s.hblk = off;
    off += al(2 * p.C * p.blk * 4, 128);
    s.hsrc = off;
    off += al(2 * p.M * p.Ec * 4, 128);
  } else {
    s.hblk = s.hsrc = -1;
  }
  s.pb = off;
  off += al(p.M * PLD * 4, 128);
  s.oc = off;
  off += al(p.Mp * p.ldo * es, 128);
  s.ac = off;                                   // end of the zero-initialised block
  off += al(p.M * p.Ec * 4, 128);
  if (cache_smem) {
    s.cs = off;
    off += al(p.U * p.M * p.Ec * es, 128);
  } else {
    s.cs = -1;
  }
  s.kvs = off;
  off += al(p.kv_slots * p.g * p.Cm * p.kvw * 4, 128);
  s.cst = off;
  off += al((p.A * p.Ec + p.Ec + p.H * p.Ec + 2 * p.E + ((p.A + 3) & ~3) + (p.headw_smem ? p.E * p.A : 0)) * 4, 128);
  s.x = off;
  off += al(p.M * p.A * 4, 16);
  s.z = off;
  off += al(p.M * p.A * 4, 16);
  s.sch = off;
  off += al(p.T * 8, 16);
  s.bars = off;
  off += (2 * p.nslot + 5) * 8;
  s.total = al(off, 128);
  p.sm = s;
  return s.total;
}

template <typename T, int MT>
static cudaError_t prepare_t(int smem_bytes, int cluster, int* max_clusters) {
  cudaError_t e = cudaFuncSetAttribute(job_kernel<T, MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  if (cluster > 8) {
    e = cudaFuncSetAttribute(job_kernel<T, MT>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(cluster, 1, 1);
  cfg.blockDim = dim3(NTHREADS, 1, 1);
  cfg.dynamicSmemBytes = smem_bytes;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  e = cudaOccupancyMaxActiveClusters(&n, job_kernel<T, MT>, &cfg);
  if (e != cudaSuccess) return e;
  *max_clusters = n;
  return cudaSuccess;
}

cudaError_t job_kernel_prepare(int dtype, int smem_bytes, int cluster, int* max_clusters) {
  // both tile-count instantiations get the attributes; the cluster count is that of the smaller one
  int n1 = 0, n2 = 0;
  cudaError_t e = dtype == 1 ? prepare_t<__nv_bfloat16, 1>(smem_bytes, cluster, &n1)
                             : prepare_t<float, 1>(smem_bytes, cluster, &n1);
  if (e != cudaSuccess) return e;
  e = dtype == 1 ? prepare_t<__nv_bfloat16, 2>(smem_bytes, cluster, &n2) : prepare_t<float, 2>(smem_bytes, cluster, &n2);
  if (e != cudaSuccess) return e;
  *max_clusters = n1 < n2 ? n1 : n2;
  return cudaSuccess;
}

template <typename T, int MT>
static cudaError_t launch_t(const JobParams& p, int n_clusters, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(n_clusters * p.C, 1, 1);
  cfg.blockDim = dim3(NTHREADS, 1, 1);
  cfg.dynamicSmemBytes = p.sm.total;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, job_kernel<T, MT>, p);
}

cudaError_t launch_job(const JobParams& p, int dtype, int n_clusters, cudaStream_t s) {
  if (p.Mp > 16)
    return dtype == 1 ? launch_t<__nv_bfloat16, 2>(p, n_clusters, s) : launch_t<float, 2>(p, n_clusters, s);
  return dtype == 1 ? launch_t<__nv_bfloat16, 1>(p, n_clusters, s) : launch_t<float, 1>(p, n_clusters, s);
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

cudaError_t launch_validate(const uint8_t* S, long long n, int* err, cudaStream_t s) {
  validate_kernel<<<1, 256, 0, s>>>(S, n, err);
  return cudaGetLastError();
}

cudaError_t launch_pop_dev(const float* x, int P, int N_obs, int HA, float* dev, cudaStream_t s) {
  pop_dev_kernel<<<P, 256, 0, s>>>(x, P, N_obs, HA, dev);
  return cudaGetLastError();
}

}  // namespace evo

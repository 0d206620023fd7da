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
// The residual stream a is distributed over the cluster by columns; each CTA
// owns E/C columns of a and of every unit's cache c_b, so a skipped cell costs
// one local add of cached values.  A refreshed unit needs two cluster
// exchanges: the CTAs all-gather a (distributed shared memory stores) to
// normalise full rows, each computes its share of the branch (attention: the
// queries/keys of its head and its slice of head dimensions; FFN: its slice
// of the hidden layer), and the second matmul's partial sums are
// reduce-scattered so that each CTA finishes its own columns.
//
// Weights never pass through registers on their way in: a producer warp per
// CTA walks the same schedule and streams, for every refreshed unit only, the
// CTA's pre-packed weight slices through a ring of shared-memory slots with
// bulk asynchronous copies (cp.async.bulk + mbarrier transaction counts).
// Skipped units generate no weight traffic, so time follows the schedule's
// refresh count.
//
// bf16 mode: GEMM operands bf16, mma.sync m16n8k16 with fp32 accumulation
// (rows per job are 16..32, far below a tcgen05 tile; the cost here is weight
// streaming and cluster latency, not tensor throughput).  fp32 mode: FFMA.
// Caches are stored in the GEMM operand type.

#include "evo_internal.h"

#include <cstdio>

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

__device__ __forceinline__ void st_cluster_v4(uint32_t addr, float4 v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(v.x), "f"(v.y), "f"(v.z),
               "f"(v.w)
               : "memory");
}

__device__ __forceinline__ void st_cluster_v2(uint32_t addr, float a, float b) {
  asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(addr), "f"(a), "f"(b) : "memory");
}

__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float a) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(a) : "memory");
}

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

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
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

// a bounded wait: after ~2 s of SM cycles the wait gives up, records
// ST_TIMEOUT and lets the thread continue so that every CTA still reaches the
// same barriers and the kernel ends.
constexpr long long WAIT_LIMIT = 4000000000LL;

struct Ctx {
  uint8_t* smem;
  uint64_t* full;
  uint64_t* empty;
  uint64_t* cbar;
  uint32_t q;      // slab counter (same sequence as the producer)
  uint32_t cph;    // cluster barrier phase parity
  int dead;
  int c, tid, warp, lane;
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

// cluster-wide barrier among the compute warps only (the producer warp runs ahead)
__device__ __forceinline__ void csync(const JobParams& p, Ctx& cx) {
  fence_cluster();
  bar_compute();
  if (cx.tid < p.C) mbar_arrive_cluster(mapa(smem_u32(cx.cbar), cx.tid));
  wait_parity(smem_u32(cx.cbar), cx.cph, true, cx, p.status);
  cx.cph ^= 1u;
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

// refresh decision for (b, t); identical in the producer and the compute warps
__device__ __forceinline__ bool refresh_of(const JobParams& p, const uint8_t* S, int b, int t, uint64_t& valid) {
  const int row = (p.S_rows == p.U) ? b : b / 3;
  const bool s = S[row * p.T + t] != 0;
  const bool v = (valid >> b) & 1ull;
  const bool r = s || (p.force && !v);
  if (r) valid |= (1ull << b);
  return r;
}

__device__ __forceinline__ int piece_K(const JobParams& p, int u, int piece) {
  return piece == 0 ? p.E : (u == 2 ? p.kp_h : p.kp_o);
}

__device__ __forceinline__ int piece_N(const JobParams& p, int u, int piece) {
  return piece == 0 ? (u == 0 ? p.n1_sa : (u == 1 ? p.n1_ca : p.n1_ff)) : p.E;
}

// ---------------------------------------------------------------------------
// producer: stream the weight slabs of refreshed units, in schedule order
// ---------------------------------------------------------------------------
template <typename T>
__device__ void producer(const JobParams& p, Ctx& cx, uint32_t cid, uint32_t ncl) {
  uint32_t q = 0;
  for (int job = cid; job < p.n_jobs; job += ncl) {
    const int s0 = min(job * p.g, p.samples - 1);
    const uint8_t* S = p.S + (long long)(s0 / p.per_sched) * p.S_stride;
    uint64_t valid = 0;
    for (int t = 0; t < p.T; ++t) {
      for (int b = 0; b < p.U; ++b) {
        if (!refresh_of(p, S, b, t, valid)) continue;
        const int l = b / 3, u = b % 3;
        for (int piece = 0; piece < 2; ++piece) {
          const int K = piece_K(p, u, piece), N = piece_N(p, u, piece);
          const uint8_t* src = p.wpack + (long long)cx.c * p.cta_stride + (long long)l * p.layer_stride +
                               p.poff[u][piece];
          const int ktb = N * 16 * (int)sizeof(T);
          const int kps = max(1, p.slot_bytes / ktb);
          const int nkt = K / 16;
          for (int kt0 = 0; kt0 < nkt; kt0 += kps) {
            const uint32_t bytes = (uint32_t)(min(kps, nkt - kt0) * ktb);
            const uint32_t slot = q % p.nslot;
            const uint32_t ph = (q / p.nslot) & 1u;
            wait_parity(smem_u32(&cx.empty[slot]), ph ^ 1u, false, cx, p.status);
            mbar_arrive_expect_tx(&cx.full[slot], bytes);
            bulk_g2s(cx.smem + p.sm.ring + slot * p.slot_bytes, src + (long long)kt0 * ktb, bytes, &cx.full[slot]);
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
// GEMM over streamed weight slabs.  A: shared memory, row-major.
// ---------------------------------------------------------------------------
template <int MT>
__device__ __forceinline__ void gemm_bf16(const JobParams& p, Ctx& cx, const __nv_bfloat16* A, int lda, int K,
                                          int N, float (&acc)[MT][8][4]) {
  const int NT = N >> 3;
  const int ntw = NT > cx.warp ? (NT - cx.warp + NCW - 1) / NCW : 0;
#pragma unroll
  for (int m = 0; m < MT; ++m)
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int r = 0; r < 4; ++r) acc[m][i][r] = 0.f;
  const int ktb = N * 32;
  const int kps = max(1, p.slot_bytes / ktb);
  const int nkt = K >> 4;
  for (int kt0 = 0; kt0 < nkt; kt0 += kps) {
    const uint8_t* slab = ring_acquire(p, cx);
    const int nk = min(kps, nkt - kt0);
    for (int kk = 0; kk < nk; ++kk) {
      uint32_t a[MT][4];
#pragma unroll
      for (int m = 0; m < MT; ++m)
        ldmatrix_x4(a[m], A + (m * 16 + (cx.lane & 15)) * lda + (kt0 + kk) * 16 + (cx.lane >> 4) * 8);
      const uint8_t* base = slab + (size_t)kk * NT * 256 + cx.lane * 8;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        if (i < ntw) {
          const int nt = cx.warp + i * NCW;
          const uint2 bf = *reinterpret_cast<const uint2*>(base + nt * 256);
#pragma unroll
          for (int m = 0; m < MT; ++m) mma_bf16(acc[m][i], a[m], bf);
        }
      }
    }
    ring_release(p, cx);
  }
}

constexpr int F32_MAXO = 16;

__device__ __forceinline__ void gemm_f32(const JobParams& p, Ctx& cx, const float* A, int lda, int K, int M, int N,
                                         float (&acc)[F32_MAXO]) {
  int mi[F32_MAXO], ni[F32_MAXO];
  const int nout = M * N;
#pragma unroll
  for (int i = 0; i < F32_MAXO; ++i) {
    const int o = cx.tid + i * NCT;
    mi[i] = o < nout ? o / N : 0;
    ni[i] = o < nout ? o % N : 0;
    acc[i] = 0.f;
  }
  const int ktb = N * 64;
  const int kps = max(1, p.slot_bytes / ktb);
  const int nkt = K >> 4;
  for (int kt0 = 0; kt0 < nkt; kt0 += kps) {
    const float* W = reinterpret_cast<const float*>(ring_acquire(p, cx));
    const int rows = min(kps, nkt - kt0) * 16;
    for (int r = 0; r < rows; ++r) {
      const int k = kt0 * 16 + r;
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

// write this CTA's columns of a into the [M][ldf] buffer `dst` of every CTA of the cluster
__device__ __forceinline__ void gather_rows(const JobParams& p, Ctx& cx, const float* ac, float* dst) {
  const uint32_t base = smem_u32(dst);
  const int nvec = p.M * p.Ec / 4;
  for (int v = cx.tid; v < nvec * p.C; v += NCT) {
    const int r = v / nvec;
    const int e = (v - r * nvec) * 4;
    const int m = e / p.Ec, j = e - m * p.Ec;
    const float4 val = *reinterpret_cast<const float4*>(ac + e);
    st_cluster_v4(mapa(base + (uint32_t)((m * p.ldf + cx.c * p.Ec + j) * 4), (uint32_t)r), val);
  }
}

// LayerNorm of full rows m < M of `buf` in place: the row is overwritten by
// its normalised values in type T (row stride in T elements = ldf * 4 / sizeof(T)).
template <typename T>
__device__ __forceinline__ void layernorm_inplace(const JobParams& p, Ctx& cx, float* buf, const float (&g)[16],
                                                  const float (&bt)[16]) {
  const int nper = p.E >> 5;
  for (int m = cx.warp; m < p.M; m += NCW) {
    float* row = buf + m * p.ldf;
    float v[16];
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (j < nper) {
        v[j] = row[cx.lane + 32 * j];
        s += v[j];
      }
    const float mean = warp_sum(s) / p.E;
    float s2 = 0.f;
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (j < nper) {
        const float d = v[j] - mean;
        s2 += d * d;
      }
    const float rstd = 1.0f / sqrtf(warp_sum(s2) / p.E + 1e-5f);
    __syncwarp();
    T* out = reinterpret_cast<T*>(row);
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (j < nper) out[cx.lane + 32 * j] = from_f<T>((v[j] - mean) * rstd * g[j] + bt[j]);
    __syncwarp();
  }
}

template <typename T>
struct Kern {
  static constexpr bool BF = sizeof(T) == 2;

  // ---- first GEMM epilogues ------------------------------------------------
  // SA / CA: f32 rows of q|k|v (SA) or q (CA) + bias;  FFN: T(gelu(. + bias))
  template <int MT>
  __device__ static void gemm1(const JobParams& p, Ctx& cx, int u, const float* bias) {
    float* xbuf = reinterpret_cast<float*>(cx.smem + p.sm.afull);
    const int N = u == 0 ? p.n1_sa : (u == 1 ? p.n1_ca : p.n1_ff);
    float* g1 = reinterpret_cast<float*>(cx.smem + p.sm.g1);
    T* hid = reinterpret_cast<T*>(cx.smem + p.sm.g1);
    if constexpr (BF) {
      float acc[MT][8][4];
      gemm_bf16<MT>(p, cx, reinterpret_cast<const __nv_bfloat16*>(xbuf), p.ldf * 2, p.E, N, acc);
      const int NT = N >> 3;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int nt = cx.warp + i * NCW;
        if (nt < NT) {
          const int n = nt * 8 + 2 * (cx.lane & 3);
          const float b0 = __ldg(bias + n), b1 = __ldg(bias + n + 1);
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int m = mt * 16 + (cx.lane >> 2) + 8 * h;
              if (m < p.M) {
                const float v0 = acc[mt][i][2 * h] + b0, v1 = acc[mt][i][2 * h + 1] + b1;
                if (u == 2) {
                  hid[m * p.ldh + n] = from_f<T>(gelu_erf(v0));
                  hid[m * p.ldh + n + 1] = from_f<T>(gelu_erf(v1));
                } else {
                  g1[m * p.ldg1 + n] = v0;
                  g1[m * p.ldg1 + n + 1] = v1;
                }
              }
            }
        }
      }
    } else {
      float acc[F32_MAXO];
      gemm_f32(p, cx, xbuf, p.ldf, p.E, p.M, N, acc);
#pragma unroll
      for (int i = 0; i < F32_MAXO; ++i) {
        const int o = cx.tid + i * NCT;
        if (o < p.M * N) {
          const int m = o / N, n = o % N;
          const float v = acc[i] + __ldg(bias + n);
          if (u == 2)
            hid[m * p.ldh + n] = from_f<T>(gelu_erf(v));
          else
            g1[m * p.ldg1 + n] = v;
        }
      }
    }
  }

  // ---- second GEMM: partial sums over this CTA's K slice, reduce-scattered
  template <int MT>
  __device__ static void gemm2(const JobParams& p, Ctx& cx, int u) {
    const T* A = reinterpret_cast<const T*>(cx.smem + (u == 2 ? p.sm.g1 : p.sm.oc));
    const int lda = u == 2 ? p.ldh : p.ldo;
    const int K = u == 2 ? p.kp_h : p.kp_o;
    const uint32_t rs = smem_u32(cx.smem + p.sm.rs);
    if constexpr (BF) {
      float acc[MT][8][4];
      gemm_bf16<MT>(p, cx, reinterpret_cast<const __nv_bfloat16*>(A), lda, K, p.E, acc);
      const int NT = p.E >> 3;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int nt = cx.warp + i * NCW;
        if (nt < NT) {
          const int n = nt * 8 + 2 * (cx.lane & 3);
          const int r = n / p.Ec, jj = n - r * p.Ec;
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int m = mt * 16 + (cx.lane >> 2) + 8 * h;
              if (m < p.M)
                st_cluster_v2(mapa(rs + (uint32_t)(((cx.c * p.M + m) * p.Ec + jj) * 4), (uint32_t)r),
                              acc[mt][i][2 * h], acc[mt][i][2 * h + 1]);
            }
        }
      }
    } else {
      float acc[F32_MAXO];
      gemm_f32(p, cx, reinterpret_cast<const float*>(A), lda, K, p.M, p.E, acc);
#pragma unroll
      for (int i = 0; i < F32_MAXO; ++i) {
        const int o = cx.tid + i * NCT;
        if (o < p.M * p.E) {
          const int m = o / p.E, n = o % p.E;
          const int r = n / p.Ec, jj = n - r * p.Ec;
          st_cluster_f32(mapa(rs + (uint32_t)(((cx.c * p.M + m) * p.Ec + jj) * 4), (uint32_t)r), acc[i]);
        }
      }
    }
  }

  // ---- attention for this CTA's head-dimension slice ------------------------
  // SA: causal over the H tokens of the same sample; q, k of the CTA's head and
  // v of its slice are in g1.  CA: keys/values of the memory tokens in kvs.
  __device__ static void attention(const JobParams& p, Ctx& cx, int u) {
    const float* g1 = reinterpret_cast<const float*>(cx.smem + p.sm.g1);
    const float* kvs = reinterpret_cast<const float*>(cx.smem + p.sm.kvs);
    T* oc = reinterpret_cast<T*>(cx.smem + p.sm.oc);
    const float scale = 1.0f / sqrtf((float)p.dh);
    const int kvw = p.dh + p.Ec;
    for (int m = cx.warp; m < p.M; m += NCW) {
      const int i = m / p.H, qi = m - i * p.H;
      const float* q = g1 + m * p.ldg1;
      const int nkey = u == 0 ? qi + 1 : p.Cm;
      float s = -INFINITY;
      if (cx.lane < nkey) {
        const float* kr = u == 0 ? g1 + (i * p.H + cx.lane) * p.ldg1 + p.dh : kvs + (i * p.Cm + cx.lane) * kvw;
        float d = 0.f;
        for (int e = 0; e < p.dh; ++e) d = fmaf(q[e], kr[e], d);
        s = d * scale;
      }
      const float mx = warp_max(s);
      const float pj = cx.lane < nkey ? expf(s - mx) : 0.f;
      const float inv = 1.0f / warp_sum(pj);
      float o0 = 0.f, o1 = 0.f;
      for (int j = 0; j < nkey; ++j) {
        const float pb = __shfl_sync(0xffffffffu, pj, j);
        const float* vr = u == 0 ? g1 + (i * p.H + j) * p.ldg1 + 2 * p.dh : kvs + (i * p.Cm + j) * kvw + p.dh;
        if (cx.lane < p.Ec) o0 = fmaf(pb, vr[cx.lane], o0);
        if (cx.lane + 32 < p.Ec) o1 = fmaf(pb, vr[cx.lane + 32], o1);
      }
      if (cx.lane < p.Ec) oc[m * p.ldo + cx.lane] = from_f<T>(o0 * inv);
      if (cx.lane + 32 < p.Ec) oc[m * p.ldo + cx.lane + 32] = from_f<T>(o1 * inv);
    }
  }

  // ---- one refreshed unit (Eq. 1, (b,t) in S) --------------------------------
  template <int MT>
  __device__ static void unit(const JobParams& p, Ctx& cx, int job, int b, int t, int sample0) {
    const int l = b / 3, u = b % 3;
    float* ac = reinterpret_cast<float*>(cx.smem + p.sm.ac);
    float* afull = reinterpret_cast<float*>(cx.smem + p.sm.afull);
    // prefetch LayerNorm parameters (lane-strided columns) and the finishing bias
    float gam[16], bet[16];
    const float* lnv = p.vec + p.v_ln + (long long)b * 2 * p.E;
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (j < (p.E >> 5)) {
        gam[j] = __ldg(lnv + cx.lane + 32 * j);
        bet[j] = __ldg(lnv + p.E + cx.lane + 32 * j);
      }
    // cross-attention: stage the memory tokens' keys (this head) and values (this slice)
    if (u == 1) {
      float* kvs = reinterpret_cast<float*>(cx.smem + p.sm.kvs);
      const int kvw = p.dh + p.Ec;
      const int h = (cx.c * p.Ec) / p.dh;
      const int kq = p.dh / 4, vq = p.Ec / 4;
      const int per_tok = kq + vq;
      const int total = p.g * p.Cm * per_tok;
      for (int v = cx.tid; v < total; v += NCT) {
        const int i = v / (p.Cm * per_tok);
        const int rem = v - i * p.Cm * per_tok;
        const int tok = rem / per_tok, w = rem - tok * per_tok;
        const int s = min(sample0 + i, p.samples - 1);
        const float* src = tok == 0 ? p.kv_time + ((long long)t * p.L + l) * 2 * p.E
                                    : p.kv_obs + (((long long)(s % p.obs_mod) * p.n_obs + (tok - 1)) * p.L + l) * 2 * p.E;
        const float* s4 = w < kq ? src + h * p.dh + 4 * w : src + p.E + cx.c * p.Ec + 4 * (w - kq);
        float* d4 = kvs + (i * p.Cm + tok) * kvw + (w < kq ? 4 * w : p.dh + 4 * (w - kq));
        cp_async16(d4, s4);
      }
    }
    bar_compute();                     // ac final for this unit
    gather_rows(p, cx, ac, afull);
    csync(p, cx);                      // exchange 1: full rows of a everywhere
    layernorm_inplace<T>(p, cx, afull, gam, bet);
    if (u == 1) cp_async_wait_all();
    bar_compute();
    gemm1<MT>(p, cx, u, p.vec + p.v_b1 + ((long long)b * p.C + cx.c) * p.n1max);
    bar_compute();
    if (u != 2) {
      attention(p, cx, u);
      bar_compute();
    }
    gemm2<MT>(p, cx, u);
    csync(p, cx);                      // exchange 2: partial sums landed
    // finish this CTA's columns: r = sum of partials + bias; c_b <- r; a += r
    const float* rs = reinterpret_cast<const float*>(cx.smem + p.sm.rs);
    T* cache = reinterpret_cast<T*>(p.cache) + ((long long)(job * p.U + b) * p.C + cx.c) * p.M * p.Ec;
    const float* b2 = p.vec + p.v_b2 + (long long)b * p.E + cx.c * p.Ec;
    for (int e = cx.tid; e < p.M * p.Ec; e += NCT) {
      const int m = e / p.Ec, j = e - m * p.Ec;
      float r = 0.f;
      for (int cc = 0; cc < p.C; ++cc) r += rs[(cc * p.M + m) * p.Ec + j];
      r += __ldg(b2 + j);
      cache[e] = from_f<T>(r);
      ac[e] += r;
      if (p.trace) {
        const int s = sample0 + m / p.H;
        if (s < p.samples)
          p.trace[(((long long)t * p.U + b) * p.samples + s) * p.H * p.E + (m % p.H) * p.E + cx.c * p.Ec + j] = r;
      }
    }
  }

  // ---- skipped unit: a += c_b on this CTA's columns ----------------------------
  __device__ static void skip_add(const JobParams& p, Ctx& cx, int job, int b, int t, int sample0, bool valid) {
    float* ac = reinterpret_cast<float*>(cx.smem + p.sm.ac);
    const T* cache = reinterpret_cast<const T*>(p.cache) + ((long long)(job * p.U + b) * p.C + cx.c) * p.M * p.Ec;
    for (int e = cx.tid; e < p.M * p.Ec; e += NCT) {
      const float cv = valid ? to_f<T>(cache[e]) : 0.f;
      if (valid) ac[e] += cv;
      if (p.trace) {
        const int m = e / p.Ec, j = e - m * p.Ec;
        const int s = sample0 + m / p.H;
        if (s < p.samples)
          p.trace[(((long long)t * p.U + b) * p.samples + s) * p.H * p.E + (m % p.H) * p.E + cx.c * p.Ec + j] = cv;
      }
    }
  }

  // ---- output head + sampler step ---------------------------------------------
  __device__ static void head_step(const JobParams& p, Ctx& cx, int t, bool any_refresh, const float (&gf)[16],
                                   const float (&bf)[16]) {
    float* ac = reinterpret_cast<float*>(cx.smem + p.sm.ac);
    float* hb = reinterpret_cast<float*>(cx.smem + (p.head_sep ? p.sm.hbuf : p.sm.afull));
    float* x = reinterpret_cast<float*>(cx.smem + p.sm.x);
    const float* z = reinterpret_cast<const float*>(cx.smem + p.sm.z);
    if (p.head_sep && !any_refresh) csync(p, cx);   // previous head's readers are done with hbuf
    bar_compute();
    gather_rows(p, cx, ac, hb);
    csync(p, cx);
    cp_async_wait_all();
    bar_compute();
    const float* tab = p.stab + t * 8;
    const float inv_sa = tab[0], s1 = tab[1], cx0 = tab[2], cxt = tab[3], sig = tab[4];
    const float sab = tab[5], sabp = tab[6], s1p = tab[7];
    const int nper = p.E >> 5;
    const float* hw = p.vec + p.v_headw;
    for (int m = cx.warp; m < p.M; m += NCW) {
      const float* row = hb + m * p.ldf;
      float v[16];
      float s = 0.f;
#pragma unroll
      for (int j = 0; j < 16; ++j)
        if (j < nper) {
          v[j] = row[cx.lane + 32 * j];
          s += v[j];
        }
      const float mean = warp_sum(s) / p.E;
      float s2 = 0.f;
#pragma unroll
      for (int j = 0; j < 16; ++j)
        if (j < nper) {
          const float d = v[j] - mean;
          s2 += d * d;
        }
      const float rstd = 1.0f / sqrtf(warp_sum(s2) / p.E + 1e-5f);
#pragma unroll
      for (int j = 0; j < 16; ++j)
        if (j < nper) v[j] = (v[j] - mean) * rstd * gf[j] + bf[j];
      float eps_mine = 0.f;
      for (int a = 0; a < p.A; ++a) {
        float part = 0.f;
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (j < nper) part = fmaf(v[j], __ldg(hw + (cx.lane + 32 * j) * p.A + a), part);
        const float e = warp_sum(part);
        if (cx.lane == a) eps_mine = e + __ldg(p.vec + p.v_headb + a);
      }
      if (cx.lane < p.A) {
        const float xv = x[m * p.A + cx.lane];
        float x0 = (xv - s1 * eps_mine) * inv_sa;
        x0 = fminf(1.0f, fmaxf(-1.0f, x0));
        float xn;
        if (p.sampler == 0) {
          xn = cx0 * x0 + cxt * xv + sig * z[m * p.A + cx.lane];
        } else {
          xn = sabp * x0 + s1p * ((xv - sab * x0) / s1);
        }
        x[m * p.A + cx.lane] = xn;
      }
    }
    if (!p.head_sep) csync(p, cx);                    // afull is rewritten by the next gather
    bar_compute();
  }

  template <int MT>
  __device__ static void compute(const JobParams& p, Ctx& cx, uint32_t cid, uint32_t ncl) {
    float* ac = reinterpret_cast<float*>(cx.smem + p.sm.ac);
    float* x = reinterpret_cast<float*>(cx.smem + p.sm.x);
    float* z = reinterpret_cast<float*>(cx.smem + p.sm.z);
    uint8_t* sch = cx.smem + p.sm.sch;
    const float* cst = reinterpret_cast<const float*>(cx.smem + p.sm.cst);
    const float* c_inw = cst;
    const float* c_inb = cst + p.A * p.Ec;
    const float* c_pos = c_inb + p.Ec;
    // per-kernel constants: LN_f parameters in registers
    float gf[16], bf[16];
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (j < (p.E >> 5)) {
        gf[j] = __ldg(p.vec + p.v_lnfg + cx.lane + 32 * j);
        bf[j] = __ldg(p.vec + p.v_lnfb + cx.lane + 32 * j);
      }
    for (int job = cid; job < p.n_jobs; job += ncl) {
      const int sample0 = job * p.g;
      const int s_first = min(sample0, p.samples - 1);
      const uint8_t* S = p.S + (long long)(s_first / p.per_sched) * p.S_stride;
      // schedule rows (expanded to units) and initial x
      for (int v = cx.tid; v < p.U * p.T; v += NCT) {
        const int b = v / p.T, t = v - b * p.T;
        const int row = (p.S_rows == p.U) ? b : b / 3;
        sch[v] = S[row * p.T + t];
      }
      for (int v = cx.tid; v < p.M * p.A; v += NCT) {
        const int m = v / p.A;
        const int s = min(sample0 + m / p.H, p.samples - 1);
        x[v] = p.noise[((long long)(s % p.obs_mod) * p.H + (m % p.H)) * p.A + (v % p.A)];
      }
      bar_compute();
      uint64_t valid = 0;
      for (int t = 0; t < p.T; ++t) {
        // stage z_t for the sampler step (DDPM)
        if (p.sampler == 0) {
          const int per = p.H * p.A / 4;
          for (int v = cx.tid; v < p.g * per; v += NCT) {
            const int i = v / per, w = v - i * per;
            const int s = min(sample0 + i, p.samples - 1);
            cp_async16(z + i * p.H * p.A + 4 * w,
                       p.noise + ((long long)(1 + t) * p.obs_mod + (s % p.obs_mod)) * p.H * p.A + 4 * w);
          }
        }
        // input embedding into this CTA's columns
        for (int e = cx.tid; e < p.M * p.Ec; e += NCT) {
          const int m = e / p.Ec, j = e - m * p.Ec;
          float acc = 0.f;
          for (int a = 0; a < p.A; ++a) acc = fmaf(x[m * p.A + a], c_inw[a * p.Ec + j], acc);
          ac[e] = acc + c_inb[j] + c_pos[(m % p.H) * p.Ec + j];
        }
        bool any = false;
        for (int b = 0; b < p.U; ++b) {
          const bool vb = (valid >> b) & 1ull;
          const bool r = sch[b * p.T + t] != 0 || (p.force && !vb);
          if (r) {
            valid |= 1ull << b;
            any = true;
            unit<MT>(p, cx, job, b, t, sample0);
          } else {
            skip_add(p, cx, job, b, t, sample0, vb);
          }
        }
        head_step(p, cx, t, any, gf, bf);
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

template <typename T>
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
  cx.q = 0;
  cx.cph = 0;
  cx.dead = 0;
  const uint32_t cid = cluster_idx(), ncl = cluster_count();

  if (threadIdx.x == 0) {
    for (int i = 0; i < p.nslot; ++i) {
      mbar_init(&cx.full[i], 1);
      mbar_init(&cx.empty[i], NCW);
    }
    mbar_init(cx.cbar, p.C);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // zero the GEMM operand buffers once: padded rows / columns must read as 0
  for (int v = threadIdx.x; v < (p.sm.ac - p.sm.afull) / 16; v += NTHREADS)
    reinterpret_cast<float4*>(smem + p.sm.afull)[v] = make_float4(0.f, 0.f, 0.f, 0.f);
  // per-kernel constant slices: in_w[:, cols], in_b[cols], pos[:, cols]
  {
    float* cst = reinterpret_cast<float*>(smem + p.sm.cst);
    const int c0 = cx.c * p.Ec;
    for (int v = threadIdx.x; v < p.A * p.Ec; v += NTHREADS)
      cst[v] = p.vec[p.v_inw + (v / p.Ec) * p.E + c0 + (v % p.Ec)];
    for (int v = threadIdx.x; v < p.Ec; v += NTHREADS) cst[p.A * p.Ec + v] = p.vec[p.v_inb + c0 + v];
    for (int v = threadIdx.x; v < p.H * p.Ec; v += NTHREADS)
      cst[p.A * p.Ec + p.Ec + v] = p.vec[p.v_pos + (v / p.Ec) * p.E + c0 + (v % p.Ec)];
  }
  __syncthreads();
  hw_cluster_sync();
  const bool bad = p.sched_err != nullptr && *p.sched_err != 0;
  if (!bad) {
    if (cx.warp == NCW) {
      if (cx.lane == 0) producer<T>(p, cx, cid, ncl);
      __syncwarp();
    } else {
      if (p.Mp > 16)
        Kern<T>::template compute<2>(p, cx, cid, ncl);
      else
        Kern<T>::template compute<1>(p, cx, cid, ncl);
    }
  }
  __syncwarp();
  hw_cluster_sync();
}

// ---------------------------------------------------------------------------
// condition path: timestep-token keys/values (once per handle) and
// observation-token keys/values (once per call)
// ---------------------------------------------------------------------------

// memory token -> per-token MLP E -> 4E (Mish) -> E, for one token per block
__device__ void cond_mlp(const float* w, const int* wo, float* tok, float* hbuf, float* out, int E) {
  const float* w1 = w + wo[W_CM_W1];
  const float* b1 = w + wo[W_CM_B1];
  const float* w2 = w + wo[W_CM_W2];
  const float* b2 = w + wo[W_CM_B2];
  __syncthreads();
  for (int j = threadIdx.x; j < 4 * E; j += blockDim.x) {
    float a = 0.f;
    for (int e = 0; e < E; ++e) a = fmaf(tok[e], w1[(long long)e * 4 * E + j], a);
    hbuf[j] = mish(a + b1[j]);
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    float a = 0.f;
    for (int j = 0; j < 4 * E; ++j) a = fmaf(hbuf[j], w2[(long long)j * E + e], a);
    out[e] = a + b2[e];
  }
  __syncthreads();
}

__device__ void memory_kv(const float* w, const int* wo, const float* mem, int L, int E, float* dst /*[L][2E]*/) {
  for (int v = threadIdx.x; v < L * 2 * E; v += blockDim.x) {
    const int l = v / (2 * E), n = v - l * 2 * E;
    const float* wl = w + wo[W_LAYER0] + (long long)l * wo[W_LAYER_STRIDE];
    const float* wkv = wl + wo[WL_CA_WKV];
    float a = 0.f;
    for (int e = 0; e < E; ++e) a = fmaf(mem[e], wkv[(long long)e * 2 * E + n], a);
    dst[v] = a + wl[wo[WL_CA_BKV] + n];
  }
}

// kv_time[t][l][2E]: keys/values of the timestep token of loop step t
__global__ void time_table_kernel(const float* w, const int* wo, const float* kstep, int L, int E, float* kv_time) {
  extern __shared__ float sh[];
  float* tok = sh;
  float* hb = sh + E;
  float* mem = hb + 4 * E;
  const int t = blockIdx.x;
  const double k = (double)kstep[t];
  const int half = E / 2;
  for (int i = threadIdx.x; i < half; i += blockDim.x) {
    const double f = exp(-log(10000.0) * (double)i / (double)(half - 1));
    tok[i] = (float)sin(k * f) + w[wo[W_COND_POS] + i];
    tok[half + i] = (float)cos(k * f) + w[wo[W_COND_POS] + half + i];
  }
  cond_mlp(w, wo, tok, hb, mem, E);
  memory_kv(w, wo, mem, L, E, kv_time + (long long)t * L * 2 * E);
}

// kv_obs[s][j][l][2E] for observation token j of sample s (one block per token)
__global__ void obs_cond_kernel(const float* w, const int* wo, const float* obs, int n_obs, int D, int L, int E,
                                float* kv_obs) {
  extern __shared__ float sh[];
  float* tok = sh;
  float* hb = sh + E;
  float* mem = hb + 4 * E;
  const int tokid = blockIdx.x;             // s * n_obs + j
  const int j = tokid % n_obs;
  const float* o = obs + (long long)tokid * D;
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    float a = 0.f;
    for (int d = 0; d < D; ++d) a = fmaf(o[d], w[wo[W_OBS_W] + (long long)d * E + e], a);
    tok[e] = a + w[wo[W_OBS_B] + e] + w[wo[W_COND_POS] + (1 + j) * E + e];
  }
  cond_mlp(w, wo, tok, hb, mem, E);
  memory_kv(w, wo, mem, L, E, kv_obs + (long long)tokid * L * 2 * E);
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
    s = warp_sum(s);
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

int smem_layout(JobParams& p, int es) {
  auto al = [](int x, int a) { return (x + a - 1) / a * a; };
  SmemLayout s{};
  int off = 0;
  s.ring = off;
  off += p.nslot * p.slot_bytes;
  s.afull = off;
  off += al(p.Mp * p.ldf * 4, 128);
  if (p.head_sep) {
    s.hbuf = off;
    off += al(p.M * p.ldf * 4, 128);
  } else {
    s.hbuf = -1;
  }
  s.rs = off;
  off += al(p.C * p.M * p.Ec * 4, 128);
  const int g1b = max(p.M * p.ldg1 * 4, p.Mp * p.ldh * es);
  s.g1 = off;
  off += al(g1b, 128);
  s.oc = off;
  off += al(p.Mp * p.ldo * es, 128);
  s.ac = off;
  off += al(p.M * p.Ec * 4, 128);
  s.kvs = off;
  off += al(p.g * p.Cm * (p.dh + p.Ec) * 4, 128);
  s.cst = off;
  off += al((p.A * p.Ec + p.Ec + p.H * p.Ec) * 4, 128);
  s.x = off;
  off += al(p.M * p.A * 4, 16);
  s.z = off;
  off += al(p.M * p.A * 4, 16);
  s.sch = off;
  off += al(p.U * p.T, 16);
  s.bars = off;
  off += (2 * p.nslot + 1) * 8;
  s.total = al(off, 128);
  p.sm = s;
  return s.total;
}

template <typename T>
static cudaError_t prepare_t(int smem_bytes, int cluster, int* max_clusters) {
  cudaError_t e = cudaFuncSetAttribute(job_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  if (cluster > 8) {
    e = cudaFuncSetAttribute(job_kernel<T>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
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
  e = cudaOccupancyMaxActiveClusters(&n, job_kernel<T>, &cfg);
  if (e != cudaSuccess) return e;
  *max_clusters = n;
  return cudaSuccess;
}

cudaError_t job_kernel_prepare(int dtype, int smem_bytes, int cluster, int* max_clusters) {
  return dtype == 1 ? prepare_t<__nv_bfloat16>(smem_bytes, cluster, max_clusters)
                    : prepare_t<float>(smem_bytes, cluster, max_clusters);
}

template <typename T>
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
  return cudaLaunchKernelEx(&cfg, job_kernel<T>, p);
}

cudaError_t launch_job(const JobParams& p, int dtype, int n_clusters, cudaStream_t s) {
  return dtype == 1 ? launch_t<__nv_bfloat16>(p, n_clusters, s) : launch_t<float>(p, n_clusters, s);
}

cudaError_t launch_time_table(const float* w, const int* wo, const float* kstep, int T, int L, int E,
                              float* kv_time, cudaStream_t s) {
  const size_t sh = (size_t)6 * E * sizeof(float);
  time_table_kernel<<<T, 256, sh, s>>>(w, wo, kstep, L, E, kv_time);
  return cudaGetLastError();
}

cudaError_t launch_obs_cond(const float* w, const int* wo, const float* obs, int N, int n_obs, int D, int L, int E,
                            float* /*unused*/, float* kv_obs, cudaStream_t s) {
  const size_t sh = (size_t)6 * E * sizeof(float);
  obs_cond_kernel<<<N * n_obs, 256, sh, s>>>(w, wo, obs, n_obs, D, L, E, kv_obs);
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

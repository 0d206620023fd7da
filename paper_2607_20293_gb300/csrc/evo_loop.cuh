// The denoising-loop kernel, compiled per model shape.
//
// One persistent kernel runs whole action queries.  A "job" is a group of G
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
// that the receiver sends once it has finished reading that buffer (argued at
// each buffer below).
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
//
// Every size below is a compile-time constant of the Shape, so the inner
// loops unroll completely and addresses fold to constants: at these sizes the
// kernel is bound by dependent latencies and control flow, not by arithmetic.
#pragma once

#include "evo_ptx.cuh"
#include "evo_shapes.h"

namespace evo {

__host__ __device__ constexpr int ct_ilog2(int x) { return x <= 1 ? 0 : 1 + ct_ilog2(x / 2); }
__host__ __device__ constexpr int ct_rup(int x, int a) { return (x + a - 1) / a * a; }
__host__ __device__ constexpr int ct_r84(int x) { return x + ((12 - x % 8) % 8); }   // smallest y >= x with y % 8 == 4
__host__ __device__ constexpr int ct_min(int a, int b) { return a < b ? a : b; }

// Model shape of one compiled loop kernel: embedding E, NH heads, horizon H,
// cluster size C, G samples per job, ES bytes per GEMM operand, ring of NSLOT
// slots of SLOT bytes.  The host plan computes the same values (checked at launch).
template <int E_, int NH_, int H_, int C_, int G_, int ES_, int SLOT_, int NSLOT_>
struct Shape {
  static constexpr int E = E_, NH = NH_, H = H_, C = C_, G = G_, ES = ES_, SLOT = SLOT_, NSLOT = NSLOT_;
  static constexpr int dh = E / NH, Ec = E / C, hid = 4 * E / C;
  static constexpr int M = G * H, MT = (M + 15) / 16, Mp = MT * 16;
  static constexpr int lEc = ct_ilog2(Ec), lH = ct_ilog2(H);
  static constexpr int blk = M * Ec + 4;
  static constexpr int lda = ES == 2 ? E + 8 : E + 4;
  static constexpr int n1_sa = 2 * dh + Ec, n1_ca = dh, n1_ff = hid;
  static constexpr int ldg1 = ct_r84(n1_sa), kvw = ct_r84(dh + Ec);
  static constexpr int kp_o = ct_rup(Ec, 16), kp_h = ct_rup(hid, 16);
  static constexpr int ldh = ES == 2 ? kp_h + 8 : kp_h, ldo = ES == 2 ? kp_o + 8 : kp_o;
  static constexpr float invE = 1.0f / E;
  __host__ __device__ static constexpr int n1(int u) { return u == 0 ? n1_sa : (u == 1 ? n1_ca : n1_ff); }
  __host__ __device__ static constexpr int hdr1(int u) { return ct_rup(n1(u) + Ec, 4) * 4; }
  // piece q of unit kind u: K x N slice behind a header, cut into ring slabs
  __host__ __device__ static constexpr int pK(int u, int q) { return q == 0 ? E : (u == 2 ? kp_h : kp_o); }
  __host__ __device__ static constexpr int pN(int u, int q) { return q == 0 ? n1(u) : E; }
  __host__ __device__ static constexpr int pHdr(int u, int q) { return q == 0 ? hdr1(u) : 0; }
  __host__ __device__ static constexpr int pKtb(int u, int q) { return 16 * pN(u, q) * ES; }
  __host__ __device__ static constexpr int pK0(int u, int q) { return ct_min((SLOT - pHdr(u, q)) / pKtb(u, q), pK(u, q) / 16); }
  __host__ __device__ static constexpr int pKps(int u, int q) { return SLOT / pKtb(u, q); }
  __host__ __device__ static constexpr int pNs(int u, int q) {
    return pK(u, q) / 16 <= pK0(u, q) ? 1 : 1 + (pK(u, q) / 16 - pK0(u, q) + pKps(u, q) - 1) / pKps(u, q);
  }
  static_assert((Ec & (Ec - 1)) == 0 && (H & (H - 1)) == 0, "Ec and H: powers of two");
  static_assert(M * Ec <= 4 * NCT, "at most four residual columns per thread");
  // slab 0 of a piece holds its header and at least one k-tile
  static_assert(pK0(0, 0) >= 1 && pK0(1, 0) >= 1 && pK0(2, 0) >= 1 && pK0(0, 1) >= 1 && pK0(2, 1) >= 1,
                "slab 0 must hold one k-tile");
};

template <typename T, class S>
struct Loop {
  static constexpr bool BF = sizeof(T) == 2;
  static constexpr int M = S::M, MT = S::MT, E = S::E, Ec = S::Ec, C = S::C, H = S::H, dh = S::dh;
  static constexpr int MEc = M * Ec;
  static constexpr int EPT = (MEc + NCT - 1) / NCT;          // residual elements per thread (1..4)
  static constexpr uint32_t XBYTES = (uint32_t)(M * E * 4);    // bytes one exchange delivers to a CTA
  // bf16 attention on the tensor cores: q, k, v of each sample staged as bf16
  // tiles (rows of LQ / LV elements) in the first GEMM's output region
  static constexpr bool MMA_ATT = BF && H % 16 == 0 && dh % 32 == 0 && Ec % 16 == 0;
  static constexpr int LQ = dh + 8, LV = Ec + 8;
  template <int U>
  __host__ __device__ static constexpr int att_keys() { return U == 0 ? H : 16; }
  template <int U>
  __host__ __device__ static constexpr int att_sample_elems() { return (H + att_keys<U>()) * LQ + att_keys<U>() * LV; }
  // bf16 GEMMs: warps 0..NWG-1 take the n-tiles (warp w: tiles w, w + NWG, ...).
  // Every warp loads the same A fragment, so NWG trades shared-memory traffic
  // per k-tile (NWG x 512 B of A + NT x 256 B of B at 128 B/cycle) against the
  // MMAs per SM sub-partition (warp w runs on w % 4, ~8 cycles per MMA).
  __host__ __device__ static constexpr int gemm_cost(int NT, int nwg) {
    const int smem = (nwg * 512 * MT + NT * 256) / 128;
    int worst = 21;                                          // one dependent MMA
    for (int s = 0; s < 4; ++s) {
      int mm = 0;
      for (int w = s; w < nwg; w += 4) mm += (NT > w ? (NT - w + nwg - 1) / nwg : 0) * MT;
      worst = worst > 8 * mm ? worst : 8 * mm;
    }
    return smem > worst ? smem : worst;
  }
  // n-tiles per warp at most max(2, those of all NCW warps): accumulators and
  // prefetched fragments fit the register file (9 warps per CTA, three share
  // one sub-partition: at most 168 registers per thread)
  __host__ __device__ static constexpr int gemm_warps_for(int NT) {
    const int cap = (NT + NCW - 1) / NCW > 2 ? (NT + NCW - 1) / NCW : 2;
    int best = NCW;
    for (int w = NCW - 1; w >= 1; --w)
      if ((NT + w - 1) / w <= cap && gemm_cost(NT, w) < gemm_cost(NT, best)) best = w;
    return best;
  }
  // (the FFN's first GEMM keeps all warps: its GELU epilogue is per tile)
  template <int U, int Q>
  __host__ __device__ static constexpr int gemm_warps() {
    return U == 2 && Q == 0 ? NCW : gemm_warps_for(S::pN(U, Q) / 8);
  }
  template <int U, int Q>
  __host__ __device__ static constexpr int gemm_ntw() { return (S::pN(U, Q) / 8 + gemm_warps<U, Q>() - 1) / gemm_warps<U, Q>(); }
  static_assert(!MMA_ATT || S::G * att_sample_elems<0>() * 2 <= S::Mp * S::lda * S::ES, "attention staging fits");
  static_assert(!MMA_ATT || S::G * att_sample_elems<1>() * 2 <= S::Mp * S::lda * S::ES, "attention staging fits");
  // With tensor-core attention the q / k / v tiles are staged in ablk, which is
  // free between LayerNorm (its last reader) and the second GEMM's staging, so
  // the first GEMM's epilogue needs no barrier after its k-loop (xln, its A
  // operand, is not overwritten).
  static_assert(!MMA_ATT || S::G * att_sample_elems<0>() * 2 <= C * S::blk * 4, "attention staging fits in ablk");
  static_assert(!MMA_ATT || S::G * att_sample_elems<1>() * 2 <= C * S::blk * 4, "attention staging fits in ablk");
  __device__ __forceinline__ static uint8_t* att_stage(const JobParams& p, Ctx& cx) {
    return cx.smem + (MMA_ATT ? p.sm.ablk : p.sm.xln);
  }

  // ---------------------------------------------------------------- rings and barriers
  // wait for the next slab not yet acquired (cx.qa); slabs are released in
  // the same order (cx.q), a warp holds at most two at a time
  __device__ __forceinline__ static const uint8_t* ring_acquire(const JobParams& p, Ctx& cx) {
    const uint32_t slot = cx.qa % S::NSLOT;
    const uint32_t ph = (cx.qa / S::NSLOT) & 1u;
    cx.qa++;
    wait_parity(smem_u32(&cx.full[slot]), ph, false, cx, p.status);
    return cx.smem + p.sm.ring + slot * S::SLOT;
  }

  __device__ __forceinline__ static void ring_release(Ctx& cx) {
    __syncwarp();
    if (cx.lane == 0) mbar_arrive(&cx.empty[cx.q % S::NSLOT]);
    cx.q++;
  }

  // cluster-wide barrier among the compute warps only (the producer warp runs
  // ahead); used where no data exchange orders a buffer's reuse
  __device__ __forceinline__ static void csync(const JobParams& p, Ctx& cx) {
    fence_cluster();
    bar_compute();
    if (cx.tid < C) mbar_arrive_cluster(mapa(smem_u32(cx.cbar), cx.tid));
    wait_parity(smem_u32(cx.cbar), cx.cph, true, cx, p.status);
    cx.cph ^= 1u;
  }

  // receive one exchange phase (`bytes` in total, XBYTES by default) on barrier `bar`
  __device__ __forceinline__ static void exchange_wait(const JobParams& p, Ctx& cx, uint64_t* bar, uint32_t& parity,
                                                       uint32_t bytes = XBYTES) {
    if (cx.tid == 0) mbar_arrive_expect_tx(bar, bytes);
    wait_parity(smem_u32(bar), parity, true, cx, p.status);
    parity ^= 1u;
  }

  // Send one block of M*Ec floats to every CTA r of the cluster: block
  // src + r*src_stride lands in CTA r at dst + c*blk (c = this CTA), counted on
  // r's barrier `rbar`.  The writers of src have executed fence_proxy_async()
  // and a bar_compute() before this call.
  __device__ __forceinline__ static void send_blocks(Ctx& cx, const float* src, int src_stride, const float* dst,
                                                     uint64_t* rbar) {
    if (cx.tid < C) {
      const uint32_t r = (uint32_t)cx.tid;
      bulk_s2c(mapa(smem_u32(dst + cx.c * S::blk), r), src + r * src_stride, (uint32_t)(MEc * 4),
               mapa(smem_u32(rbar), r));
    }
  }

  // Send `bytes` from src to every CTA r of the cluster, landing at dst (this
  // CTA's slot in r's buffer, same offset in every CTA), counted on r's
  // barrier `rbar`; the C copies are issued by lanes of different warps.  The
  // writers of src have executed fence_proxy_async() and a bar_compute().
  // (with src_stride > 0, CTA r gets src + r * src_stride bytes instead)
  __device__ __forceinline__ static void send_spread(Ctx& cx, const void* src, uint32_t bytes, const void* dst,
                                                     uint64_t* rbar, uint32_t src_stride = 0) {
    constexpr int PER = (C + NCW - 1) / NCW;
    const int r = cx.warp + NCW * cx.lane;
    if (cx.lane < PER && r < C)
      bulk_s2c(mapa(smem_u32(dst), (uint32_t)r), reinterpret_cast<const uint8_t*>(src) + r * src_stride, bytes,
               mapa(smem_u32(rbar), (uint32_t)r));
  }

  // ---------------------------------------------------------------- producer warp
  // The whole warp turns the job's lattice into one refresh mask per step (its
  // own copy, psch); lane 0 then walks the refreshed units in order and streams
  // their weight slabs through the ring.
  __device__ __forceinline__ static void producer(const JobParams& p, Ctx& cx, uint32_t cid, uint32_t ncl) {
    uint64_t* psch = reinterpret_cast<uint64_t*>(cx.smem + p.sm.psch);
    const uint64_t units = p.U >= 64 ? ~0ull : (1ull << p.U) - 1ull;
    uint32_t q = 0;
    for (int job = cid; job < p.n_jobs; job += ncl) {
      const int s0 = min(job * S::G, p.samples - 1);
      const uint8_t* Sl = p.S + (long long)(s0 / p.per_sched) * p.S_stride;
      for (int t = cx.lane; t < p.T; t += 32) {
        uint64_t mask = 0;
#pragma unroll 8
        for (int b = 0; b < p.U; ++b) {
          const int row = (p.S_rows == p.U) ? b : b / 3;
          if (Sl[row * p.T + t] != 0) mask |= 1ull << b;
        }
        psch[t] = mask;
      }
      __syncwarp();
      uint64_t valid = 0;
      for (int t = 0; t < p.T && cx.lane == 0; ++t) {
        uint64_t refresh = (psch[t] | (p.force ? ~valid : 0ull)) & units;   // same rule as the compute warps
        valid |= refresh;
        while (refresh) {
          const int b = __ffsll((long long)refresh) - 1;
          refresh &= refresh - 1ull;
          const int l = b / 3, u = b % 3;
          for (int piece = 0; piece < 2; ++piece) {
            const uint8_t* src =
                p.wpack + (long long)cx.c * p.cta_stride + (long long)l * p.layer_stride + p.poff[u][piece];
            const int ns = S::pNs(u, piece), k0 = S::pK0(u, piece), kps = S::pKps(u, piece);
            const int ktb = S::pKtb(u, piece), hdr = S::pHdr(u, piece), nkt = S::pK(u, piece) / 16;
            for (int s = 0; s < ns; ++s) {
              const int kt0 = s == 0 ? 0 : k0 + (s - 1) * kps;
              const int cnt = s == 0 ? k0 : min(kps, nkt - kt0);
              const uint32_t off = s == 0 ? 0u : (uint32_t)(hdr + kt0 * ktb);
              const uint32_t bytes = (uint32_t)((s == 0 ? hdr : 0) + cnt * ktb);
              const uint32_t slot = q % S::NSLOT;
              const uint32_t ph = (q / S::NSLOT) & 1u;
              if (!mbar_try_wait(smem_u32(&cx.empty[slot]), ph ^ 1u)) {
                // the producer runs ahead of the compute warps: poll gently
                const long long t0 = clock64();
                while (!cx.dead && !mbar_try_wait(smem_u32(&cx.empty[slot]), ph ^ 1u)) {
                  __nanosleep(64);
                  if (clock64() - t0 > cx.wait_limit) {
                    atomicOr(p.status, ST_TIMEOUT);
                    cx.dead = 1;
                  }
                }
              }
              mbar_arrive_expect_tx(&cx.full[slot], bytes);
              bulk_g2s(cx.smem + p.sm.ring + slot * S::SLOT, src + off, bytes, &cx.full[slot]);
              ++q;
            }
          }
        }
      }
      __syncwarp();
    }
    if (cx.lane != 0) return;
    // drain: every slab issued has landed before this CTA may exit (bounded waits)
    const uint32_t first = q > (uint32_t)S::NSLOT ? q - S::NSLOT : 0u;
    for (uint32_t k = first; k < q; ++k)
      wait_parity(smem_u32(&cx.full[k % S::NSLOT]), (k / S::NSLOT) & 1u, false, cx, p.status);
  }

  // ---------------------------------------------------------------- GEMMs over streamed slabs
  // Piece (U, Q) arrives as NS slabs: slab 0 holds the header and k-tiles
  // 0..K0-1, slab s >= 1 the next KPS k-tiles.  The slab boundaries are
  // compile-time, so in the unrolled k-loop each warp waits for slab s at its
  // first k-tile and releases it after its last one: the producer refills a
  // slot as soon as every warp is past it, and a piece may span more slabs
  // than the ring has slots.
  template <int U, int Q>
  __device__ __forceinline__ static constexpr bool slab_first(int kt) {
    return kt >= S::pK0(U, Q) && (kt - S::pK0(U, Q)) % S::pKps(U, Q) == 0;
  }
  template <int U, int Q>
  __device__ __forceinline__ static constexpr bool slab_last(int kt) {
    return kt == S::pK(U, Q) / 16 - 1 || slab_first<U, Q>(kt + 1);
  }

  // bf16: warp w < NWG owns n-tiles w, w + NWG, ... (NTW of them).  The A and B
  // fragments of k-tile kt + PD are loaded right after the MMAs of k-tile kt,
  // PD k-tiles ahead of their use, so shared-memory latency and slab waits
  // overlap the MMA chain; a slab is acquired when its first k-tile is loaded
  // and released after its last k-tile's MMAs.  With
  // PD = 2 a load window spans at most two slabs unless a middle slab holds a
  // single k-tile (then PD = 1).
  template <int U, int Q>
  __device__ __forceinline__ static void gemm_bf16(const JobParams& p, Ctx& cx, const __nv_bfloat16* A, int lda,
                                                   const uint8_t* slab0, float (&acc)[MT][gemm_ntw<U, Q>()][4]) {
    constexpr int NT = S::pN(U, Q) / 8, NWG = gemm_warps<U, Q>(), NTW = gemm_ntw<U, Q>();
    constexpr int NKT = S::pK(U, Q) / 16, K0 = S::pK0(U, Q), KPS = S::pKps(U, Q);
    constexpr int HDR = S::pHdr(U, Q);
    constexpr int PD = (KPS >= 2 || NKT <= K0 + 1) ? 2 : 1, NB = PD + 1;
    static_assert(S::NSLOT >= 2, "prefetch holds two slabs");
    if (NWG < NCW && cx.warp >= NWG) {                  // warps without tiles only pass the slabs on
#pragma unroll
      for (int kt = 0; kt < NKT; ++kt) {
        if (slab_first<U, Q>(kt)) ring_acquire(p, cx);
        if (slab_last<U, Q>(kt)) ring_release(cx);
      }
      return;
    }
    const uint8_t* sl = slab0 + HDR + cx.lane * 8;
#pragma unroll
    for (int m = 0; m < MT; ++m)
#pragma unroll
      for (int i = 0; i < NTW; ++i)
#pragma unroll
        for (int r = 0; r < 4; ++r) acc[m][i][r] = 0.f;
    const __nv_bfloat16* arow = A + (cx.lane & 15) * lda + (cx.lane >> 4) * 8;
    uint32_t af[NB][MT][4];
    uint2 bf[NB][NTW];
    auto load = [&](const int kt) {
      if (slab_first<U, Q>(kt)) sl = ring_acquire(p, cx) + cx.lane * 8;
      const int kk = kt < K0 ? kt : (kt - K0) % KPS;
#pragma unroll
      for (int m = 0; m < MT; ++m) ldmatrix_x4(af[kt % NB][m], arow + m * 16 * lda + kt * 16);
#pragma unroll
      for (int i = 0; i < NTW; ++i) {
        const int nt = cx.warp + i * NWG;
        if (NT % NWG == 0 || nt < NT) bf[kt % NB][i] = *reinterpret_cast<const uint2*>(sl + (kk * NT + nt) * 256);
      }
    };
#pragma unroll
    for (int kt = 0; kt < PD; ++kt)
      if (kt < NKT) load(kt);
#pragma unroll
    for (int kt = 0; kt < NKT; ++kt) {
#pragma unroll
      for (int i = 0; i < NTW; ++i) {
        const int nt = cx.warp + i * NWG;
        if (NT % NWG == 0 || nt < NT) {
#pragma unroll
          for (int m = 0; m < MT; ++m) mma_bf16(acc[m][i], af[kt % NB][m], bf[kt % NB][i]);
        }
      }
      if (slab_last<U, Q>(kt)) ring_release(cx);
      if (kt + PD < NKT) load(kt + PD);          // after the MMAs: a slab wait overlaps them
    }
  }

  // fp32: one output per thread and slot i (M*N <= 16*NCT)
  static constexpr int F32_MAXO = 16;
  template <int U, int Q>
  __device__ __forceinline__ static void gemm_f32(const JobParams& p, Ctx& cx, const float* A, int lda,
                                                  const uint8_t* slab0, float (&acc)[F32_MAXO]) {
    constexpr int N = S::pN(U, Q), NKT = S::pK(U, Q) / 16, K0 = S::pK0(U, Q), KPS = S::pKps(U, Q);
    constexpr int HDR = S::pHdr(U, Q);
    constexpr int NOUT = M * N;
    constexpr int NO = (NOUT + NCT - 1) / NCT;
    static_assert(NO <= F32_MAXO, "fp32 GEMM: at most 16 outputs per thread");
    const float* sl = reinterpret_cast<const float*>(slab0 + HDR);
#pragma unroll
    for (int i = 0; i < F32_MAXO; ++i) acc[i] = 0.f;
#pragma unroll
    for (int kt = 0; kt < NKT; ++kt) {
      if (slab_first<U, Q>(kt)) sl = reinterpret_cast<const float*>(ring_acquire(p, cx));
      const int r0 = (kt < K0 ? kt : (kt - K0) % KPS) * 16;
#pragma unroll 4
      for (int k = 0; k < 16; ++k) {
#pragma unroll
        for (int i = 0; i < NO; ++i) {
          const int o = cx.tid + i * NCT;
          if (NOUT % NCT == 0 || o < NOUT)
            acc[i] = fmaf(A[(o / N) * lda + kt * 16 + k], sl[(r0 + k) * N + (o % N)], acc[i]);
        }
      }
      if (slab_last<U, Q>(kt)) ring_release(cx);
    }
  }

  // ---------------------------------------------------------------- LayerNorm
  // Rows m < M, half a warp per row, one pass for the mean and the second
  // moment.  Row m is read from the gathered blocks (column col is in block
  // col/Ec) and written to the A operand xln in type T.
  // In bf16 mode the gathered blocks hold bf16 (block c at c * 2blk elements).
  // The affine (gain, shift) is folded into the first GEMM's weights and bias.
  __device__ __forceinline__ static void layernorm_rows(Ctx& cx, const float* blk, T* xln) {
    constexpr int NV = E / 64;
    const int half = cx.lane >> 4, hl = cx.lane & 15;
#pragma unroll
    for (int m0 = 0; m0 < M; m0 += 2 * NCW) {
      const int m = m0 + cx.warp * 2 + half;
      if (M % (2 * NCW) == 0 || m0 + cx.warp * 2 < M) {
        float4 v[NV];
        float s = 0.f, s2 = 0.f;
#pragma unroll
        for (int j = 0; j < NV; ++j) {
          const int col = 4 * (hl + 16 * j);
          if constexpr (BF) {
            const uint2 raw = *reinterpret_cast<const uint2*>(reinterpret_cast<const __nv_bfloat16*>(blk) +
                                                              (col >> S::lEc) * (2 * S::blk) + (m << S::lEc) +
                                                              (col & (Ec - 1)));
            const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&raw.x));
            const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&raw.y));
            v[j] = make_float4(lo.x, lo.y, hi.x, hi.y);
          } else {
            v[j] = *reinterpret_cast<const float4*>(blk + (col >> S::lEc) * S::blk + (m << S::lEc) + (col & (Ec - 1)));
          }
          s += (v[j].x + v[j].y) + (v[j].z + v[j].w);
          s2 += (v[j].x * v[j].x + v[j].y * v[j].y) + (v[j].z * v[j].z + v[j].w * v[j].w);
        }
#pragma unroll
        for (int o = 8; o > 0; o >>= 1) {
          s += __shfl_xor_sync(0xffffffffu, s, o);
          s2 += __shfl_xor_sync(0xffffffffu, s2, o);
        }
        const float mean = s * S::invE;
        const float rstd = rsqrtf(fmaxf(s2 * S::invE - mean * mean, 0.f) + 1e-5f);
#pragma unroll
        for (int j = 0; j < NV; ++j) {
          const int col = 4 * (hl + 16 * j);
          const float y0 = (v[j].x - mean) * rstd, y1 = (v[j].y - mean) * rstd;
          const float y2 = (v[j].z - mean) * rstd, y3 = (v[j].w - mean) * rstd;
          T* dst = xln + m * S::lda + col;
          if constexpr (BF) {
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
  }

  __device__ __forceinline__ static T* cache_ptr(const JobParams& p, Ctx& cx, int job, int b) {
    if (p.sm.cs >= 0) return reinterpret_cast<T*>(cx.smem + p.sm.cs) + b * MEc;
    return reinterpret_cast<T*>(p.cache) + ((long long)(job * p.U + b) * C + cx.c) * MEc;
  }

  // ---------------------------------------------------------------- first GEMM
  // A = xln.  SA / CA: q|k|v (SA) or q (CA) + bias, as bf16 attention tiles in
  // ablk (tensor-core attention) or f32 rows aliasing xln; FFN:
  // T(gelu(. + bias)) aliasing xln.  Where the output aliases xln, all warps
  // finish their k-loop before any epilogue writes.
  template <int U>
  __device__ __forceinline__ static void gemm1(const JobParams& p, Ctx& cx, const uint8_t* slab0) {
    constexpr int N = S::n1(U);
    const float* bias = reinterpret_cast<const float*>(slab0);
    float* g1 = reinterpret_cast<float*>(cx.smem + p.sm.xln);
    T* hid = reinterpret_cast<T*>(cx.smem + p.sm.xln);
    if constexpr (BF) {
      constexpr int NT = N / 8, NWG = gemm_warps<U, 0>(), NTW = gemm_ntw<U, 0>();
      float2 bv[NTW];
#pragma unroll
      for (int i = 0; i < NTW; ++i) {
        const int nt = cx.warp + i * NWG;
        bv[i] = (cx.warp < NWG && (NT % NWG == 0 || nt < NT))
                    ? *reinterpret_cast<const float2*>(bias + nt * 8 + 2 * (cx.lane & 3))
                    : make_float2(0.f, 0.f);
      }
      float acc[MT][NTW][4];
      gemm_bf16<U, 0>(p, cx, reinterpret_cast<const __nv_bfloat16*>(cx.smem + p.sm.xln), S::lda, slab0, acc);
      if constexpr (!(MMA_ATT && U != 2)) bar_compute();     // the output aliases xln
#pragma unroll
      for (int i = 0; i < NTW; ++i) {
        const int nt = cx.warp + i * NWG;
        if (cx.warp < NWG && (NT % NWG == 0 || nt < NT)) {
          const int n = nt * 8 + 2 * (cx.lane & 3);
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int m = mt * 16 + (cx.lane >> 2) + 8 * h;
              if (M % 16 == 0 || m < M) {
                const float v0 = acc[mt][i][2 * h] + bv[i].x, v1 = acc[mt][i][2 * h + 1] + bv[i].y;
                if constexpr (U == 2) {
                  *reinterpret_cast<__nv_bfloat162*>(hid + m * S::ldh + n) =
                      __floats2bfloat162_rn(gelu_as(v0), gelu_as(v1));
                } else if constexpr (MMA_ATT) {
                  // q -> Q[i], k -> K[i], v -> V[i] of sample m / H
                  __nv_bfloat16* st = reinterpret_cast<__nv_bfloat16*>(att_stage(p, cx)) +
                                      (m >> S::lH) * att_sample_elems<U>();
                  const int i = m & (H - 1);
                  __nv_bfloat16* dst = n < dh       ? st + i * LQ + n
                                       : n < 2 * dh ? st + (H + i) * LQ + (n - dh)
                                                    : st + (H + att_keys<U>()) * LQ + i * LV + (n - 2 * dh);
                  *reinterpret_cast<__nv_bfloat162*>(dst) = __floats2bfloat162_rn(v0, v1);
                } else {
                  *reinterpret_cast<float2*>(g1 + m * S::ldg1 + n) = make_float2(v0, v1);
                }
              }
            }
        }
      }
    } else {
      constexpr int NOUT = M * N, NO = (NOUT + NCT - 1) / NCT;
      float bv[F32_MAXO];
#pragma unroll
      for (int i = 0; i < F32_MAXO; ++i) {
        const int o = cx.tid + i * NCT;
        bv[i] = (i < NO && o < NOUT) ? bias[o % N] : 0.f;
      }
      float acc[F32_MAXO];
      gemm_f32<U, 0>(p, cx, reinterpret_cast<const float*>(cx.smem + p.sm.xln), S::lda, slab0, acc);
      bar_compute();
#pragma unroll
      for (int i = 0; i < NO; ++i) {
        const int o = cx.tid + i * NCT;
        if (o < NOUT) {
          const int m = o / N, n = o % N;
          const float v = acc[i] + bv[i];
          if constexpr (U == 2)
            hid[m * S::ldh + n] = from_f<T>(gelu_as(v));
          else
            g1[m * S::ldg1 + n] = v;
        }
      }
    }
  }

  // ---------------------------------------------------------------- second GEMM
  // Partial sums over this CTA's K slice, staged in ablk in block layout
  // (block r = columns r*Ec.. destined for CTA r; in bf16 mode as bf16 in the
  // first half of the block).  Staging into ablk is safe
  // block by block: CTA r's next gather writes only block r of ablk, and r can
  // only send it after it has received this CTA's partial block r.
  template <int U>
  __device__ __forceinline__ static void gemm2(const JobParams& p, Ctx& cx, const uint8_t* slab0) {
    const T* A = reinterpret_cast<const T*>(cx.smem + (U == 2 ? p.sm.xln : p.sm.oc));
    constexpr int lda = U == 2 ? S::ldh : S::ldo;
    float* stage = reinterpret_cast<float*>(cx.smem + p.sm.ablk);
    if constexpr (BF) {
      constexpr int NT = E / 8, NWG = gemm_warps<U, 1>(), NTW = gemm_ntw<U, 1>();
      float acc[MT][NTW][4];
      gemm_bf16<U, 1>(p, cx, reinterpret_cast<const __nv_bfloat16*>(A), lda, slab0, acc);
#pragma unroll
      for (int i = 0; i < NTW; ++i) {
        const int nt = cx.warp + i * NWG;
        if (cx.warp < NWG && (NT % NWG == 0 || nt < NT)) {
          const int n = nt * 8 + 2 * (cx.lane & 3);
          __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(stage + (n >> S::lEc) * S::blk) + (n & (Ec - 1));
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int m = mt * 16 + (cx.lane >> 2) + 8 * h;
              if (M % 16 == 0 || m < M)
                *reinterpret_cast<__nv_bfloat162*>(dst + (m << S::lEc)) =
                    __floats2bfloat162_rn(acc[mt][i][2 * h], acc[mt][i][2 * h + 1]);
            }
        }
      }
    } else {
      constexpr int NOUT = M * E, NO = (NOUT + NCT - 1) / NCT;
      float acc[F32_MAXO];
      gemm_f32<U, 1>(p, cx, reinterpret_cast<const float*>(A), lda, slab0, acc);
#pragma unroll
      for (int i = 0; i < NO; ++i) {
        const int o = cx.tid + i * NCT;
        if (o < NOUT) {
          const int m = o / E, n = o % E;
          stage[(n >> S::lEc) * S::blk + (m << S::lEc) + (n & (Ec - 1))] = acc[i];
        }
      }
    }
  }

  // ---------------------------------------------------------------- attention
  // Scores: one (query row, key) pair per thread, softmax over groups of G
  // lanes (G = keys rounded up to a power of two), probabilities to pb; then
  // one output (row, dim of this CTA's slice) per thread.  SA: causal over the
  // H tokens of the same sample (q, k of the CTA's head and v of its slice are
  // rows of the first GEMM's output).  CA: the 1 + n_obs memory tokens in kvs.
  // Tensor-core attention (bf16): warp s < G takes sample s.  S = Q K^T
  // (mma.sync m16n8k16), causal (SA) or key-count (CA, memory tokens padded
  // to 16) mask and softmax on the accumulators, O = P V with P taken from
  // the score registers; O goes to the second GEMM's A operand.
  template <int U>
  __device__ __forceinline__ static void attention_mma(const JobParams& p, Ctx& cx, const float* kvs) {
    constexpr int NK = att_keys<U>(), NKT = NK / 8, MTH = H / 16;
    if (cx.warp >= S::G) return;
    const int sm_ = cx.warp, lane = cx.lane;
    __nv_bfloat16* Q = reinterpret_cast<__nv_bfloat16*>(att_stage(p, cx)) + sm_ * att_sample_elems<U>();
    __nv_bfloat16* K = Q + H * LQ;
    __nv_bfloat16* V = K + NK * LQ;
    const int g = lane >> 2, tq = lane & 3;
    float sc[MTH][NKT][4];
#pragma unroll
    for (int m = 0; m < MTH; ++m)
#pragma unroll
      for (int n = 0; n < NKT; ++n) sc[m][n][0] = sc[m][n][1] = sc[m][n][2] = sc[m][n][3] = 0.f;
#pragma unroll
    for (int k2 = 0; k2 < dh / 32; ++k2) {
      uint32_t a0[MTH][4], a1[MTH][4];
#pragma unroll
      for (int m = 0; m < MTH; ++m) {
        const __nv_bfloat16* qa = Q + (m * 16 + (lane & 15)) * LQ + k2 * 32 + (lane >> 4) * 8;
        ldmatrix_x4(a0[m], qa);
        ldmatrix_x4(a1[m], qa + 16);
      }
#pragma unroll
      for (int n = 0; n < NKT; ++n) {
        uint32_t b[4];
        ldmatrix_x4(b, K + (n * 8 + (lane & 7)) * LQ + k2 * 32 + (lane >> 3) * 8);
#pragma unroll
        for (int m = 0; m < MTH; ++m) {
          mma_bf16(sc[m][n], a0[m], make_uint2(b[0], b[1]));
          mma_bf16(sc[m][n], a1[m], make_uint2(b[2], b[3]));
        }
      }
    }
    const float scale = rsqrtf((float)dh);
    const int nkeys = U == 0 ? H : p.Cm;
    float inv[MTH][2];
#pragma unroll
    for (int m = 0; m < MTH; ++m) {
      float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
      for (int n = 0; n < NKT; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int row = m * 16 + g + (e >> 1) * 8, col = n * 8 + 2 * tq + (e & 1);
          const bool keep = U == 0 ? col <= row : col < nkeys;
          const float v = keep ? sc[m][n][e] * scale : -INFINITY;
          sc[m][n][e] = v;
          mx[e >> 1] = fmaxf(mx[e >> 1], v);
        }
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        mx[hh] = fmaxf(mx[hh], __shfl_xor_sync(0xffffffffu, mx[hh], 1));
        mx[hh] = fmaxf(mx[hh], __shfl_xor_sync(0xffffffffu, mx[hh], 2));
      }
      float sum[2] = {0.f, 0.f};
#pragma unroll
      for (int n = 0; n < NKT; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float v = sc[m][n][e] == -INFINITY ? 0.f : __expf(sc[m][n][e] - mx[e >> 1]);
          sc[m][n][e] = v;
          sum[e >> 1] += v;
        }
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        sum[hh] += __shfl_xor_sync(0xffffffffu, sum[hh], 1);
        sum[hh] += __shfl_xor_sync(0xffffffffu, sum[hh], 2);
        inv[m][hh] = __frcp_rn(sum[hh]);
      }
    }
    float o[MTH][Ec / 8][4];
#pragma unroll
    for (int m = 0; m < MTH; ++m)
#pragma unroll
      for (int n = 0; n < Ec / 8; ++n) o[m][n][0] = o[m][n][1] = o[m][n][2] = o[m][n][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < NK / 16; ++kk) {
      uint32_t a[MTH][4];
#pragma unroll
      for (int m = 0; m < MTH; ++m) {
        __nv_bfloat162 h0 = __floats2bfloat162_rn(sc[m][2 * kk][0], sc[m][2 * kk][1]);
        __nv_bfloat162 h1 = __floats2bfloat162_rn(sc[m][2 * kk][2], sc[m][2 * kk][3]);
        __nv_bfloat162 h2 = __floats2bfloat162_rn(sc[m][2 * kk + 1][0], sc[m][2 * kk + 1][1]);
        __nv_bfloat162 h3 = __floats2bfloat162_rn(sc[m][2 * kk + 1][2], sc[m][2 * kk + 1][3]);
        a[m][0] = *reinterpret_cast<uint32_t*>(&h0);
        a[m][1] = *reinterpret_cast<uint32_t*>(&h1);
        a[m][2] = *reinterpret_cast<uint32_t*>(&h2);
        a[m][3] = *reinterpret_cast<uint32_t*>(&h3);
      }
#pragma unroll
      for (int n2 = 0; n2 < Ec / 16; ++n2) {
        uint32_t b[4];
        ldmatrix_x4_trans(b, V + (kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * LV + n2 * 16 + (lane >> 4) * 8);
#pragma unroll
        for (int m = 0; m < MTH; ++m) {
          mma_bf16(o[m][2 * n2], a[m], make_uint2(b[0], b[1]));
          mma_bf16(o[m][2 * n2 + 1], a[m], make_uint2(b[2], b[3]));
        }
      }
    }
    T* oc = reinterpret_cast<T*>(cx.smem + p.sm.oc);
#pragma unroll
    for (int m = 0; m < MTH; ++m)
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        T* dst = oc + (sm_ * H + m * 16 + g + hh * 8) * S::ldo + 2 * tq;
#pragma unroll
        for (int n = 0; n < Ec / 8; ++n)
          *reinterpret_cast<__nv_bfloat162*>(dst + n * 8) =
              __floats2bfloat162_rn(o[m][n][2 * hh] * inv[m][hh], o[m][n][2 * hh + 1] * inv[m][hh]);
      }
  }

  // memory keys / values of every sample of the job (fp32 in kvs) -> the bf16
  // K / V tiles of the cross-attention, padded keys zero; all compute threads
  __device__ __forceinline__ static void stage_memory_kv(const JobParams& p, Ctx& cx, const float* kvs) {
    constexpr int NK = att_keys<1>(), PK = NK * (dh / 2), PS = NK * ((dh + Ec) / 2);
    for (int c = cx.tid; c < S::G * PS; c += NCT) {
      const int s_ = c / PS, r = c - s_ * PS;
      __nv_bfloat16* K = reinterpret_cast<__nv_bfloat16*>(att_stage(p, cx)) + s_ * att_sample_elems<1>() + H * LQ;
      const float* kv = kvs + s_ * p.Cm * S::kvw;
      const bool isk = r < PK;
      const int j = isk ? r / (dh / 2) : (r - PK) / (Ec / 2);
      const int d = isk ? 2 * (r % (dh / 2)) : 2 * ((r - PK) % (Ec / 2));
      const float2 f =
          j < p.Cm ? *reinterpret_cast<const float2*>(kv + j * S::kvw + (isk ? 0 : dh) + d) : make_float2(0.f, 0.f);
      __nv_bfloat16* dst = isk ? K + j * LQ + d : K + NK * LQ + j * LV + d;
      *reinterpret_cast<__nv_bfloat162*>(dst) = __floats2bfloat162_rn(f.x, f.y);
    }
  }

  template <int U>
  __device__ __forceinline__ static void attention(const JobParams& p, Ctx& cx, const float* kvs) {
    if constexpr (MMA_ATT) {
      if constexpr (U == 1) {
        stage_memory_kv(p, cx, kvs);
        bar_compute();
      }
      attention_mma<U>(p, cx, kvs);
      return;
    }
    const float* g1 = reinterpret_cast<const float*>(cx.smem + p.sm.xln);
    float* pb = reinterpret_cast<float*>(cx.smem + p.sm.pb);
    T* oc = reinterpret_cast<T*>(cx.smem + p.sm.oc);
    const float scale = rsqrtf((float)dh);
    const int nk = U == 0 ? H : p.Cm;
    int lG = 0;
    while ((1 << lG) < nk) ++lG;
    const int G = 1 << lG;
    const int rows_per_pass = NCT >> lG;
    for (int base = 0; base < M; base += rows_per_pass) {
      const int m = base + (cx.tid >> lG), j = cx.tid & (G - 1);
      float s = -INFINITY;
      const bool live = m < M && j < nk;
      if (live) {
        const int i = m >> S::lH, qi = m & (H - 1);
        if (U != 0 || j <= qi) {
          const float4* q4 = reinterpret_cast<const float4*>(g1 + m * S::ldg1);
          const float4* k4 = U == 0 ? reinterpret_cast<const float4*>(g1 + ((i << S::lH) + j) * S::ldg1 + dh)
                                    : reinterpret_cast<const float4*>(kvs + (i * p.Cm + j) * S::kvw);
          float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
#pragma unroll
          for (int e = 0; e < dh / 4; ++e) {
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
      const float ex = s == -INFINITY ? 0.f : __expf(s - mx);
      const float sum = group_sum_dyn(ex, G);
      if (live) pb[m * PLD + j] = ex * __frcp_rn(sum);
    }
    bar_compute();
#pragma unroll
    for (int k = 0; k < EPT; ++k) {
      const int o = cx.tid + k * NCT;
      if (MEc % NCT == 0 || o < MEc) {
        const int m = o >> S::lEc, e = o & (Ec - 1);
        const int i = m >> S::lH, qi = m & (H - 1);
        const float* prow = pb + m * PLD;
        float a0 = 0.f, a1 = 0.f;
        if constexpr (U == 0) {
          const float* v = g1 + (i << S::lH) * S::ldg1 + 2 * dh + e;
#pragma unroll
          for (int j = 0; j < H; j += 2) {
            if (j <= qi) a0 = fmaf(prow[j], v[j * S::ldg1], a0);
            if (j + 1 <= qi) a1 = fmaf(prow[j + 1], v[(j + 1) * S::ldg1], a1);
          }
        } else {
          const float* v = kvs + (i * p.Cm) * S::kvw + dh + e;
          for (int j = 0; j < p.Cm; ++j) a0 = fmaf(prow[j], v[j * S::kvw], a0);
        }
        oc[m * S::ldo + e] = from_f<T>(a0 + a1);
      }
    }
  }

  // stage the memory tokens' keys (this CTA's head) and values (its slice) of
  // layer l at step t into kvs (cp.async; waited before use)
  __device__ __forceinline__ static void stage_kv(const JobParams& p, Ctx& cx, int l, int t, float* kvs) {
    if (cx.kv_i >= 0) {
      const float* src = cx.kv_base + (cx.kv_tok == 0 ? (long long)t * p.L * 2 * E : 0ll) + l * 2 * E + cx.kv_src;
      cp_async16(kvs + cx.kv_dst, src);
    }
  }

  // per-job part of the staging map (which sample's observation rows this thread copies)
  __device__ __forceinline__ static void stage_kv_job(const JobParams& p, Ctx& cx, int sample0) {
    if (cx.kv_i < 0) return;
    const int s = min(sample0 + cx.kv_i, p.samples - 1);
    cx.kv_base = cx.kv_tok == 0 ? p.kv_time
                                : p.kv_obs + ((long long)(s % p.obs_mod) * p.n_obs + (cx.kv_tok - 1)) * p.L * 2 * E;
  }

  // ---------------------------------------------------------------- one refreshed unit (Eq. 1, (b,t) in S)
  // bnext: the next refreshed unit of this step (U if none); the finish adds
  // the cached outputs of b+1..bnext-1 and, when bnext < U, prepares its gather.
  template <int U>
  __device__ __forceinline__ static void unit(const JobParams& p, Ctx& cx, int job, int b, int t, int sample0,
                                              int bnext) {
    const int l = b / 3;
    float* ac = reinterpret_cast<float*>(cx.smem + p.sm.ac);
    float* ablk = reinterpret_cast<float*>(cx.smem + p.sm.ablk);
    float* kvs = reinterpret_cast<float*>(cx.smem + p.sm.kvs);
    if constexpr (U == 1) {
      if (p.kv_slots == 1) stage_kv(p, cx, l, t, kvs);
      else kvs += l * S::G * p.Cm * S::kvw;
    }
    // exchange 1: every CTA receives every CTA's columns of a (rounded to bf16
    // in bf16 mode: they are only LayerNorm's input, whose output is bf16).
    // ablk is read by LayerNorm below; CTA r sends into it again only after
    // this CTA's partial sums (sent after the first GEMM) reached r.
    // slab 0 of piece 1 ([first bias | second-GEMM bias slice | k-tiles]) is
    // acquired while the exchange is in flight
    const uint8_t* s1;
    if constexpr (BF) {
      __nv_bfloat16* acb = reinterpret_cast<__nv_bfloat16*>(cx.smem + p.sm.acb);   // written by the preceding pass
      fence_proxy_async();
      bar_compute();                   // ac final for this unit
      send_spread(cx, acb, (uint32_t)(MEc * 2), ablk + cx.c * S::blk, cx.xg);
      s1 = ring_acquire(p, cx);
      exchange_wait(p, cx, cx.xg, cx.pg, XBYTES / 2);
    } else {
      fence_proxy_async();
      bar_compute();                   // ac final for this unit
      send_blocks(cx, ac, 0, ablk, cx.xg);
      s1 = ring_acquire(p, cx);
      exchange_wait(p, cx, cx.xg, cx.pg);
    }
    const float* hdr = reinterpret_cast<const float*>(s1);
    float b2[EPT];
#pragma unroll
    for (int k = 0; k < EPT; ++k) b2[k] = hdr[S::n1(U) + ((cx.tid + k * NCT) & (Ec - 1))];
    layernorm_rows(cx, ablk, reinterpret_cast<T*>(cx.smem + p.sm.xln));
    bar_compute();
    gemm1<U>(p, cx, s1);
    const uint8_t* s2 = ring_acquire(p, cx);      // slab 0 of piece 2, held through the attention
    if constexpr (U == 1) cp_async_wait_all();
    bar_compute();
    if constexpr (U != 2) {
      attention<U>(p, cx, kvs);
      bar_compute();
    }
    gemm2<U>(p, cx, s2);
    // exchange 2: block r of the staged partial sums goes to CTA r (bf16 in
    // bf16 mode).  rs is read below; CTA r sends into it again only after this
    // CTA's next gather.
    fence_proxy_async();
    bar_compute();
    const float* rs = reinterpret_cast<const float*>(cx.smem + p.sm.rs);
    if constexpr (BF) {
      send_spread(cx, ablk, (uint32_t)(MEc * 2), rs + cx.c * S::blk, cx.xr, (uint32_t)(S::blk * 4));
      exchange_wait(p, cx, cx.xr, cx.pr, XBYTES / 2);
    } else {
      send_blocks(cx, ablk, S::blk, rs, cx.xr);
      exchange_wait(p, cx, cx.xr, cx.pr);
    }
    // finish this CTA's columns: r = sum of partials + bias; c_b <- r; a += r
    T* cache = cache_ptr(p, cx, job, b);
#pragma unroll
    for (int k = 0; k < EPT; ++k) {
      const int e = cx.tid + k * NCT;
      if (MEc % NCT == 0 || e < MEc) {
        float part[C];
#pragma unroll
        for (int cc = 0; cc < C; ++cc)
          part[cc] = BF ? to_f<__nv_bfloat16>(reinterpret_cast<const __nv_bfloat16*>(rs + cc * S::blk)[e])
                        : rs[cc * S::blk + e];
#pragma unroll
        for (int w = C / 2; w > 0; w >>= 1)
#pragma unroll
          for (int cc = 0; cc < w; ++cc) part[cc] += part[cc + w];
        const float r = part[0] + b2[k];
        cache[e] = from_f<T>(r);
        if (p.trace) {
          const int m = e >> S::lEc, j = e & (Ec - 1);
          const int s = sample0 + (m >> S::lH);
          if (s < p.samples && dcheck(t < p.T && b < p.U && cx.c * Ec + j < E, p.status))
            p.trace[(((long long)t * p.U + b) * p.samples + s) * H * E + (m & (H - 1)) * E + cx.c * Ec + j] = r;
        }
        const float a = add_cached(p, cx, job, b + 1, bnext, t, sample0, e, ac[e] + r);
        ac[e] = a;
        if (BF && bnext < p.U) reinterpret_cast<__nv_bfloat16*>(cx.smem + p.sm.acb)[e] = __float2bfloat16_rn(a);
      }
    }
  }

  // ---------------------------------------------------------------- skipped units b0..b1-1 (Eq. 1: a += c_b)
  // Element e of this CTA's columns: a + the cached outputs of the skipped
  // units b0..b1-1 (zero for a unit not refreshed yet in this query), loaded
  // eight at a time and summed pairwise before the add.  Runs inside the
  // per-element pass that precedes them (the embedding or a refreshed unit's
  // finish).
  __device__ __forceinline__ static float add_cached(const JobParams& p, Ctx& cx, int job, int b0, int b1, int t,
                                                     int sample0, int e, float a) {
    if (b0 >= b1) return a;
    const int cstride = p.sm.cs >= 0 ? MEc : C * MEc;
    const T* cb = cache_ptr(p, cx, job, b0) + e;
    for (int b = b0; b < b1; b += 8, cb += 8 * cstride) {
      const int n = b1 - b;                           // uniform over the block
      float cv[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) cv[q] = q < n ? to_f<T>(cb[q * cstride]) : 0.f;
      a += ((cv[0] + cv[1]) + (cv[2] + cv[3])) + ((cv[4] + cv[5]) + (cv[6] + cv[7]));
      if (p.trace) {
        const int m = e >> S::lEc, j = e & (Ec - 1);
        const int s = sample0 + (m >> S::lH);
        if (s < p.samples) {
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (b + q < b1)
              p.trace[(((long long)t * p.U + b + q) * p.samples + s) * H * E + (m & (H - 1)) * E + cx.c * Ec + j] =
                  cv[q];
        }
      }
    }
    return a;
  }

  // ---------------------------------------------------------------- output head + sampler step
  // eps = LN_f(a) W_head + b_head (Eq. 1's denoiser output) from per-row partial
  // sums: with mean, rstd of the full row, (LN_f(a) W)_a = rstd (sum_e a_e g_e W_ea
  // - mean G_a) + B_a, G_a = sum_e g_e W_ea, B_a = sum_e b_e W_ea.  Each CTA
  // reduces its own columns to 2 + A numbers per row (sum, sum of squares, the
  // A dots with gw = g W) and all-gathers them; every CTA then adds the C
  // partials of each row in the same order, so all CTAs hold the same x.
  // Without head_sep the blocks land in ablk at c*blk: block c of CTA r last
  // held r's second-GEMM partials for this CTA, which this CTA has received.
  __device__ __forceinline__ static void head_step(const JobParams& p, Ctx& cx, int t) {
    const float* ac = reinterpret_cast<const float*>(cx.smem + p.sm.ac);
    float* x = reinterpret_cast<float*>(cx.smem + p.sm.x);
    const float* z = reinterpret_cast<const float*>(cx.smem + p.sm.z);
    const float* cst = reinterpret_cast<const float*>(cx.smem + p.sm.cst);
    const int A4 = (p.A + 3) & ~3, NP = 2 + p.A, npr = p.npr;
    const float* head_b = cst + p.A * Ec + Ec + H * Ec;
    const float* Gs = head_b + A4;
    const float* Bs = head_b + 2 * A4;
    const float* gw = head_b + 3 * A4;
    const int par = p.head_sep ? (t & 1) : 0;
    float* ps = reinterpret_cast<float*>(cx.smem + p.sm.hsrc) + par * M * npr;
    const int hstr = p.head_sep ? M * npr : S::blk;   // landing stride between the C blocks
    const float* hb = reinterpret_cast<const float*>(cx.smem + p.sm.hblk) + par * C * M * npr;
    // 1. this CTA's partials.  Up to 16 columns: one element per thread, reduced
    //    over the Ec lanes of its row with shuffles; more columns: thread
    //    o < M * NP takes quantity q of row m as one dot product over the
    //    columns (a . 1, a . a, a . gw[q - 2]).  (Measured: the first is faster
    //    on 16 columns, the second on 64.)
    if constexpr (Ec <= 16) {
#pragma unroll
      for (int k = 0; k < EPT; ++k) {
        const int e = cx.tid + k * NCT;
        if (MEc % NCT == 0 || e < MEc) {         // MEc is a multiple of 64: warp-uniform
          const int m = e >> S::lEc, j = e & (Ec - 1);
          const bool lead = j == 0;
          float* dst = ps + m * npr;
          const float v = ac[e];
          float s0 = v, s1 = v * v;
#pragma unroll
          for (int o = Ec / 2; o > 0; o >>= 1) {
            s0 += __shfl_xor_sync(0xffffffffu, s0, o);
            s1 += __shfl_xor_sync(0xffffffffu, s1, o);
          }
          if (lead) {
            dst[0] = s0;
            dst[1] = s1;
          }
          for (int a = 0; a < p.A; ++a) {
            float d = v * gw[a * Ec + j];
#pragma unroll
            for (int o = Ec / 2; o > 0; o >>= 1) d += __shfl_xor_sync(0xffffffffu, d, o);
            if (lead) dst[2 + a] = d;
          }
        }
      }
    } else {
      // a thread reads a whole row of ac, written element by element by other
      // threads (the last refreshed unit's finish, or the step's embedding)
      bar_compute();
      for (int o = cx.tid; o < M * NP; o += NCT) {
        const int m = o / NP, q = o - m * NP;
        const float* arow = ac + m * Ec;
        const float* wrow = gw + (q >= 2 ? q - 2 : 0) * Ec;
        float acc = 0.f;
#pragma unroll
        for (int j = 0; j < Ec; ++j) {
          const float a = arow[j];
          acc = fmaf(a, q == 0 ? 1.f : (q == 1 ? a : wrow[j]), acc);
        }
        ps[m * npr + q] = acc;
      }
    }
    cp_async_wait_all();                 // z_t (issued after the previous step's head)
    fence_proxy_async();
    bar_compute();
    // 2. all-gather: the block of M*npr floats to every CTA, issue spread over the warps
    send_spread(cx, ps, (uint32_t)(M * npr * 4), hb + cx.c * hstr, cx.xh + par);
    exchange_wait(p, cx, cx.xh + par, par ? cx.ph1 : cx.ph0, (uint32_t)(C * M * npr * 4));
    // 3. rows: half a warp per row; lane hl adds quantity hl (and hl + 16) over the partials
    const float4 tab0 = *reinterpret_cast<const float4*>(cx.smem + p.sm.stb + t * 32);
    const float4 tab1 = *reinterpret_cast<const float4*>(cx.smem + p.sm.stb + t * 32 + 16);
    const float inv_sa = tab0.x, s1c = tab0.y, cx0 = tab0.z, cxt = tab0.w, sig = tab1.x;
    const float sab = tab1.y, sabp = tab1.z, s1p = tab1.w;
    const int half = cx.lane >> 4, hl = cx.lane & 15;
#pragma unroll
    for (int m0 = 0; m0 < M; m0 += 2 * NCW) {
      if (M % (2 * NCW) == 0 || m0 + cx.warp * 2 < M) {
        const int m = m0 + cx.warp * 2 + half;
        float t0 = 0.f, t1 = 0.f;
        if constexpr (Ec <= 16) {                 // (measured faster on 16 partials)
#pragma unroll
          for (int r = 0; r < C; ++r) {
            const float* src = hb + r * hstr + m * npr;
            if (hl < NP) t0 += src[hl];
            if (hl + 16 < NP) t1 += src[hl + 16];
          }
        } else {
          float v0[C], v1[C];
#pragma unroll
          for (int r = 0; r < C; ++r) {
            const float* src = hb + r * hstr + m * npr;
            v0[r] = hl < NP ? src[hl] : 0.f;
            v1[r] = hl + 16 < NP ? src[hl + 16] : 0.f;
          }
#pragma unroll
          for (int w = C / 2; w > 0; w >>= 1)
#pragma unroll
            for (int r = 0; r < w; ++r) {
              v0[r] += v0[r + w];
              v1[r] += v1[r + w];
            }
          t0 = v0[0];
          t1 = v1[0];
        }
        const float S0 = __shfl_sync(0xffffffffu, t0, 0, 16);
        const float S1 = __shfl_sync(0xffffffffu, t0, 1, 16);
        const int qd = 2 + hl;
        const float d0 = __shfl_sync(0xffffffffu, t0, qd & 15, 16);
        const float d1 = __shfl_sync(0xffffffffu, t1, qd & 15, 16);
        if (hl < p.A) {
          const float D = qd < 16 ? d0 : d1;
          const float mean = S0 * S::invE;
          const float rstd = rsqrtf(fmaxf(S1 * S::invE - mean * mean, 0.f) + 1e-5f);
          const float eps = rstd * (D - mean * Gs[hl]) + Bs[hl] + head_b[hl];
          const float xv = x[m * p.A + hl];
          float x0 = (xv - s1c * eps) * inv_sa;
          x0 = fminf(1.0f, fmaxf(-1.0f, x0));
          float xn;
          if (p.sampler == 0) {
            xn = cx0 * x0 + cxt * xv + sig * z[m * p.A + hl];
          } else {
            xn = sabp * x0 + s1p * ((xv - sab * x0) / s1c);
          }
          x[m * p.A + hl] = xn;
        }
      }
    }
    if (!p.head_sep) csync(p, cx);                    // one landing buffer: every CTA has read it
    bar_compute();
  }

  // ---------------------------------------------------------------- the compute warps' job loop
  __device__ __forceinline__ static void compute(const JobParams& p, Ctx& cx, uint32_t cid, uint32_t ncl) {
    float* ac = reinterpret_cast<float*>(cx.smem + p.sm.ac);
    float* x = reinterpret_cast<float*>(cx.smem + p.sm.x);
    float* z = reinterpret_cast<float*>(cx.smem + p.sm.z);
    uint64_t* sch = reinterpret_cast<uint64_t*>(cx.smem + p.sm.sch);
    float* kvs = reinterpret_cast<float*>(cx.smem + p.sm.kvs);
    const float* cst = reinterpret_cast<const float*>(cx.smem + p.sm.cst);
    const float* c_inw = cst;
    const float* c_inb = cst + p.A * Ec;
    const float* c_pos = c_inb + Ec;
    for (int job = cid; job < p.n_jobs; job += ncl) {
      const int sample0 = job * S::G;
      const int s_first = min(sample0, p.samples - 1);
      const uint8_t* Sl = p.S + (long long)(s_first / p.per_sched) * p.S_stride;
      // the job's lattice as one refresh mask per step, and the initial x
      for (int t = cx.tid; t < p.T; t += NCT) {
        uint64_t mask = 0;
        for (int b = 0; b < p.U; ++b) {
          const int row = (p.S_rows == p.U) ? b : b / 3;
          if (Sl[row * p.T + t] != 0) mask |= 1ull << b;
        }
        sch[t] = mask;
      }
      for (int v = cx.tid; v < M * p.A; v += NCT) {
        const int m = v / p.A;
        const int s = min(sample0 + (m >> S::lH), p.samples - 1);
        x[v] = p.noise[((long long)(s % p.obs_mod) * H + (m & (H - 1))) * p.A + (v % p.A)];
      }
      stage_kv_job(p, cx, sample0);
      // the job's caches start as zero tensors: under the zero policy a unit not
      // yet refreshed adds nothing (Sec. 3.1 cache reset), so the skip adds need no mask
      for (int b = 0; b < p.U; ++b) {
        T* cb = cache_ptr(p, cx, job, b);
        for (int e = cx.tid; e < MEc; e += NCT) cb[e] = from_f<T>(0.f);
      }
      // DDPM noise: thread v < G*H*A/4 copies 16 bytes of z_t per step (one chunk per thread)
      const float* zsrc = nullptr;
      int zdst = 0;
      if (p.sampler == 0) {
        const int per = H * p.A / 4;
        if (cx.tid < S::G * per) {
          const int i = cx.tid / per, w = cx.tid - i * per;
          const int s = min(sample0 + i, p.samples - 1);
          zsrc = p.noise + ((long long)p.obs_mod + (s % p.obs_mod)) * H * p.A + 4 * w;   // slot 1 + t at t = 0
          zdst = i * H * p.A + 4 * w;
        }
      }
      const long long zstep = (long long)p.obs_mod * H * p.A;
      if (zsrc) cp_async16(z + zdst, zsrc);                      // z_0
      const uint64_t units = p.U >= 64 ? ~0ull : (1ull << p.U) - 1ull;
      constexpr uint64_t CA_UNITS = 0x2492492492492492ull;     // bits 3l + 1: cross-attention units
      bar_compute();
      uint64_t valid = 0;
      for (int t = 0; t < p.T; ++t) {
        const uint64_t refresh = (sch[t] | (p.force ? ~valid : 0ull)) & units;
        // when every layer has a slot, stage the memory keys/values of this
        // step's refreshed cross-attention units
        if (p.kv_slots > 1)
          for (uint64_t ca = refresh & CA_UNITS; ca; ca &= ca - 1ull) {
            const int l = (__ffsll((long long)ca) - 1) / 3;
            stage_kv(p, cx, l, t, kvs + l * S::G * p.Cm * S::kvw);
          }
        // input embedding into this CTA's columns, plus the cached outputs of the
        // skipped units before the first refreshed one
        int b = refresh ? __ffsll((long long)refresh) - 1 : p.U;
#pragma unroll
        for (int k = 0; k < EPT; ++k) {
          const int e = cx.tid + k * NCT;
          if (MEc % NCT == 0 || e < MEc) {
            const int m = e >> S::lEc, j = e & (Ec - 1);
            float acc = 0.f;
            for (int a = 0; a < p.A; ++a) acc = fmaf(x[m * p.A + a], c_inw[a * Ec + j], acc);
            const float a = add_cached(p, cx, job, 0, b, t, sample0, e, acc + c_inb[j] + c_pos[(m & (H - 1)) * Ec + j]);
            ac[e] = a;
            if (BF && b < p.U) reinterpret_cast<__nv_bfloat16*>(cx.smem + p.sm.acb)[e] = __float2bfloat16_rn(a);
          }
        }
        // refreshed units in order; each finish adds the skipped units up to the next one
        while (b < p.U) {
          valid |= 1ull << b;
          const uint64_t later = b + 1 < 64 ? refresh >> (b + 1) : 0ull;
          const int bnext = later ? b + __ffsll((long long)later) : p.U;
          const int u = b % 3;
          if (u == 0) unit<0>(p, cx, job, b, t, sample0, bnext);
          else if (u == 1) unit<1>(p, cx, job, b, t, sample0, bnext);
          else unit<2>(p, cx, job, b, t, sample0, bnext);
          b = bnext;
        }
        head_step(p, cx, t);
        // DDPM noise of the next step (every thread has read z_t: head_step ends with a barrier)
        if (zsrc && t + 1 < p.T) cp_async16(z + zdst, zsrc + (t + 1) * zstep);
      }
      // write the finished chunk
      if (cx.c == 0) {
        for (int v = cx.tid; v < M * p.A; v += NCT) {
          const int s = sample0 + v / (H * p.A);
          if (s < p.samples && dcheck((long long)sample0 * H * p.A + v < (long long)p.samples * H * p.A, p.status))
            p.out[(long long)sample0 * H * p.A + v] = x[v];
        }
      }
      bar_compute();
    }
  }
};

template <typename T, class S>
__global__ void __launch_bounds__(NTHREADS, 1) job_kernel(const __grid_constant__ JobParams p) {
  extern __shared__ __align__(128) uint8_t smem[];
  Ctx cx;
  cx.smem = smem;
  cx.tid = threadIdx.x;
  cx.warp = threadIdx.x >> 5;
  cx.lane = threadIdx.x & 31;
  cx.c = (int)cluster_ctarank();
  cx.full = reinterpret_cast<uint64_t*>(smem + p.sm.bars);
  cx.empty = cx.full + S::NSLOT;
  cx.cbar = cx.full + 2 * S::NSLOT;
  cx.xg = cx.cbar + 1;
  cx.xr = cx.cbar + 2;
  cx.xh = cx.cbar + 3;
  cx.q = cx.qa = 0;
  cx.cph = cx.pg = cx.pr = cx.ph0 = cx.ph1 = 0;
  cx.dead = 0;
  cx.wait_limit = p.wait_limit;
  {
    // staging map: chunk v = tid over [G][1+n_obs][k chunks (dh/4) | v chunks (Ec/4)]
    constexpr int kq = S::dh / 4, per_tok = kq + S::Ec / 4;
    const int v = threadIdx.x;
    cx.kv_i = -1;
    cx.kv_base = nullptr;
    if (v < S::G * p.Cm * per_tok) {
      const int i = v / (p.Cm * per_tok);
      const int rem = v - i * p.Cm * per_tok;
      const int tok = rem / per_tok, w = rem - tok * per_tok;
      const int head = (cx.c * S::Ec) / S::dh;
      cx.kv_i = i;
      cx.kv_tok = tok;
      cx.kv_src = w < kq ? head * S::dh + 4 * w : S::E + cx.c * S::Ec + 4 * (w - kq);
      cx.kv_dst = (i * p.Cm + tok) * S::kvw + (w < kq ? 4 * w : S::dh + 4 * (w - kq));
    }
  }
  const uint32_t cid = cluster_idx(), ncl = cluster_count();

  if (threadIdx.x == 0) {
    for (int i = 0; i < S::NSLOT; ++i) {
      mbar_init(&cx.full[i], 1);
      mbar_init(&cx.empty[i], NCW);
    }
    mbar_init(cx.cbar, S::C);
    mbar_init(cx.xg, 1);
    mbar_init(cx.xr, 1);
    mbar_init(cx.xh, 1);
    mbar_init(cx.xh + 1, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // zero the operand and exchange buffers once: padded rows and columns must read as 0
  for (int v = threadIdx.x; v < (p.sm.ac - p.sm.ablk) / 16; v += NTHREADS)
    reinterpret_cast<float4*>(smem + p.sm.ablk)[v] = make_float4(0.f, 0.f, 0.f, 0.f);
  // sampler coefficients of every step
  for (int v = threadIdx.x; v < p.T * 8; v += NTHREADS) reinterpret_cast<float*>(smem + p.sm.stb)[v] = p.stab[v];
  // per-kernel constants: in_w[:, cols], in_b[cols], pos[:, cols], lnf_g, lnf_b, head_b, head_w
  {
    float* cst = reinterpret_cast<float*>(smem + p.sm.cst);
    const int c0 = cx.c * S::Ec;
    for (int v = threadIdx.x; v < p.A * S::Ec; v += NTHREADS)
      cst[v] = p.vec[p.v_inw + (v / S::Ec) * S::E + c0 + (v % S::Ec)];
    float* d = cst + p.A * S::Ec;
    for (int v = threadIdx.x; v < S::Ec; v += NTHREADS) d[v] = p.vec[p.v_inb + c0 + v];
    d += S::Ec;
    for (int v = threadIdx.x; v < S::H * S::Ec; v += NTHREADS)
      d[v] = p.vec[p.v_pos + (v / S::Ec) * S::E + c0 + (v % S::Ec)];
    d += S::H * S::Ec;
    const int A4 = (p.A + 3) & ~3;
    for (int v = threadIdx.x; v < p.A; v += NTHREADS) {
      d[v] = p.vec[p.v_headb + v];
      d[A4 + v] = p.vec[p.v_headG + v];
      d[2 * A4 + v] = p.vec[p.v_headB + v];
    }
    d += 3 * A4;
    for (int v = threadIdx.x; v < p.A * S::Ec; v += NTHREADS) {   // gw[a][j] = lnf_g[col] * W_head[col][a]
      const int a = v / S::Ec, col = c0 + v % S::Ec;
      d[v] = p.vec[p.v_lnfg + col] * p.vec[p.v_headw + (long long)a * S::E + col];
    }
  }
  __syncthreads();
  hw_cluster_sync();
  const bool bad = p.sched_err != nullptr && *p.sched_err != 0;
  if (!bad) {
    if (cx.warp == NCW) {
      Loop<T, S>::producer(p, cx, cid, ncl);
      __syncwarp();
    } else {
      Loop<T, S>::compute(p, cx, cid, ncl);
    }
  }
  __syncwarp();
  hw_cluster_sync();
  // In normal operation every exchange copy has been waited for by its
  // receiver before the receiver arrives here, and a sender arrives only
  // after its own waits, so no copy is in flight once all CTAs have passed
  // this barrier.  After a timeout a CTA skips its remaining waits, so the
  // last copies may still be landing (cluster barriers do not order the
  // asynchronous copies): give them time before the shared memory is freed.
  settle_after_timeout(p.status, cx.dead != 0);
}

// Host side of one shape: the plan must agree with the compile-time constants.
template <typename T, class S>
bool shape_matches(const JobParams& p) {
  return p.E == S::E && p.dh == S::dh && p.H == S::H && p.C == S::C && p.g == S::G && p.M == S::M &&
         p.Mp == S::Mp && p.blk == S::blk && p.lda == S::lda && p.ldg1 == S::ldg1 && p.kvw == S::kvw &&
         p.ldh == S::ldh && p.ldo == S::ldo && p.kp_o == S::kp_o && p.kp_h == S::kp_h && p.nslot == S::NSLOT &&
         p.slot_bytes == S::SLOT && p.hdr1[0] == S::hdr1(0) && p.hdr1[1] == S::hdr1(1) && p.hdr1[2] == S::hdr1(2) &&
         (int)sizeof(T) == S::ES;
}

template <typename T, class S>
cudaError_t shape_prepare(int smem_bytes, int* max_clusters) {
  // The limit is a process-wide attribute of the kernel: allow the device
  // maximum, so that handles with different plans of this shape coexist (each
  // launch passes its own size).
  int dev = 0, optin = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(job_kernel<T, S>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           optin > smem_bytes ? optin : smem_bytes);
  if (e != cudaSuccess) return e;
  if (S::C > 8) {
    e = cudaFuncSetAttribute(job_kernel<T, S>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S::C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(S::C, 1, 1);
  cfg.blockDim = dim3(NTHREADS, 1, 1);
  cfg.dynamicSmemBytes = smem_bytes;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaOccupancyMaxActiveClusters(max_clusters, job_kernel<T, S>, &cfg);
}

template <typename T, class S>
cudaError_t shape_launch(const JobParams& p, int n_clusters, cudaStream_t s) {
  if (!shape_matches<T, S>(p)) return cudaErrorInvalidConfiguration;   // host plan and compiled shape disagree
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S::C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(n_clusters * S::C, 1, 1);
  cfg.blockDim = dim3(NTHREADS, 1, 1);
  cfg.dynamicSmemBytes = p.sm.total;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, job_kernel<T, S>, p);
}

template <int ID>
struct ShapeOf;
EVO_SHAPES(EVO_SHAPE_SPEC)

}  // namespace evo

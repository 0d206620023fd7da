// Internal declarations shared by the host API (evo_api.cu) and the kernels
// (evo_job.cu).  Not part of the C ABI.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <vector>

#include "evo.h"

namespace evo {

constexpr int NCW = 8;              // compute warps per CTA
constexpr int NCT = NCW * 32;       // compute threads per CTA
constexpr int NTHREADS = NCT + 32;  // + one weight-streaming (producer) warp
constexpr int MAX_CLUSTER = 16;
constexpr int PLD = 33;             // row stride (floats) of the attention-probability buffer

// error bits written to the device status word
constexpr int ST_SCHEDULE = 1;
constexpr int ST_TIMEOUT = 2;
constexpr int ST_INDEX = 4;         // a device-side index check failed (debug builds)

// Device-side index checks of the debug build (EVO_DEBUG_CHECKS): a failed
// check records ST_INDEX in the status word and the caller skips the access
// (no trap, so the context stays usable).  In the normal build it is a
// constant true and costs nothing.
#ifdef EVO_DEBUG_CHECKS
__device__ __forceinline__ bool dcheck(bool ok, int* status) {
  if (!ok) atomicOr(status, ST_INDEX);
  return ok;
}
#else
__device__ __forceinline__ constexpr bool dcheck(bool, int*) { return true; }
#endif

// Guard bands around the activation buffers: GUARD_BYTES of a fixed pattern
// before and after each one, so that a kernel writing past either end is
// caught by evo_check_guards (a stand-in for a memory checker).
constexpr size_t GUARD_BYTES = 4096;
constexpr unsigned char GUARD_FILL = 0xA7;
struct GuardedRegion {
  unsigned char* base;   // allocation start: [guard | user bytes | guard]
  size_t bytes;          // user bytes
};
using GuardList = std::vector<GuardedRegion>;
// cudaMalloc of bytes + 2 guards; *user = the first byte after the leading guard
cudaError_t guarded_malloc(void** user, size_t bytes, GuardList* list);
void guarded_free(void* user);
// 0: every guard intact; 1: a guard was overwritten; -1: a CUDA call failed
int guards_check(const GuardList& list);

// Limits of the bounded waits (kernel parameters, so that a diagnostic can run
// the same helpers with a tiny limit): the loop kernel gives up after this many
// SM cycles (~2 s), the tensor-core kernels after this many polls.
constexpr long long WAIT_CYCLES_DEFAULT = 4000000000LL;
constexpr long long WAIT_POLLS_DEFAULT = 1ll << 26;
// After a wait gave up, copies issued by other threads or CTAs may still be in
// flight into this CTA's shared memory (or reading from it): before the CTA
// exits it gives them this many cycles (~0.2 ms) to land.
constexpr long long SETTLE_CYCLES = 400000LL;

__device__ __forceinline__ void settle_after_timeout(const int* status, bool dead) {
  if (!dead && !(*reinterpret_cast<const volatile int*>(status) & ST_TIMEOUT)) return;
  const long long t0 = clock64();
  while (clock64() - t0 < SETTLE_CYCLES) __nanosleep(1000);
}

// fp32 arithmetic with subnormal inputs and results flushed to zero, scalar and
// packed in pairs (one f32x2 instruction for two values; each half rounds and
// flushes exactly like the scalar operation).
__device__ __forceinline__ float fma_z(float a, float b, float c) {
  float d;
  asm("fma.rn.ftz.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
__device__ __forceinline__ float mul_z(float a, float b) {
  float d;
  asm("mul.rn.ftz.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
  return d;
}
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rc, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n mov.b64 rc, {%6, %7};\n"
      " fma.rn.ftz.f32x2 rd, ra, rb, rc;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
      " mul.rn.ftz.f32x2 rd, ra, rb;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
// exact IEEE addition (no flush): the bias adds of the GEMM epilogues
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
      " add.rn.f32x2 rd, ra, rb;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ float ex2_approx(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
// max(x, 0) that keeps NaN
__device__ __forceinline__ float relu_nan(float x) {
  float r;
  asm("max.NaN.f32 %0, %1, 0f00000000;" : "=f"(r) : "f"(x));
  return r;
}

// The erf-form GELU of the feed-forward units, x·Φ(x) = ½x(1 + erf(x/√2)),
// with erf from Abramowitz & Stegun, Handbook of Mathematical Functions,
// formula 7.1.26 (Hastings' rational form): for z ≥ 0
//   erf z = 1 − (a1 t + a2 t² + a3 t³ + a4 t⁴ + a5 t⁵) e^(−z²) + ε,  t = 1/(1 + p z),
// |ε| ≤ 1.5e-7.  With z = |x|/√2 and h = ½|x|·(1 − erf z) ≥ 0 the unit is
// max(x, 0) − h (one fused multiply-add).  |x| is capped at 16 inside h, where e^(−z²) has long
// underflowed to 0, so ±inf give inf / 0 and NaN stays NaN; subnormal
// intermediates (|x| beyond ~13, or subnormal x) flush to zero, an absolute
// change below 1e-37.  One reciprocal and one base-2 exponential on the
// special-function unit.  gelu_as2 evaluates two values with packed f32x2
// arithmetic, rounding and flushing exactly as gelu_as does.
namespace gelu_k {
constexpr float P = 0.3275911f * 0.70710678118654752f;                       // p / √2
constexpr float A1 = 0.5f * 0.254829592f, A2 = 0.5f * -0.284496736f, A3 = 0.5f * 1.421413741f,
                A4 = 0.5f * -1.453152027f, A5 = 0.5f * 1.061405429f;          // ½ a_i
constexpr float C = -0.72134752044448170f;                                    // −log2(e) / 2
constexpr float XMAX = 16.f;
}  // namespace gelu_k

__device__ __forceinline__ float gelu_as(float x) {
  using namespace gelu_k;
  const float ax = fminf(fabsf(x), XMAX);
  const float t = rcp_approx(fma_z(P, ax, 1.f));
  const float g = ex2_approx(mul_z(ax, mul_z(ax, C)));                          // e^(−x²/2)
  float q = fma_z(t, A5, A4);
  q = fma_z(t, q, A3);
  q = fma_z(t, q, A2);
  q = fma_z(t, q, A1);
  const float w = mul_z(mul_z(t, q), g);                                        // ½(1 − erf z)
  return fma_z(-ax, w, relu_nan(x));                                            // max(x, 0) − |x| w, one rounding
}

__device__ __forceinline__ float2 gelu_as2(float2 x) {
  using namespace gelu_k;
  const float2 ax = make_float2(fminf(fabsf(x.x), XMAX), fminf(fabsf(x.y), XMAX));
  const float2 u = fma2(make_float2(P, P), ax, make_float2(1.f, 1.f));
  const float2 t = make_float2(rcp_approx(u.x), rcp_approx(u.y));
  const float2 s = mul2(ax, mul2(ax, make_float2(C, C)));
  const float2 g = make_float2(ex2_approx(s.x), ex2_approx(s.y));
  float2 q = fma2(t, make_float2(A5, A5), make_float2(A4, A4));
  q = fma2(t, q, make_float2(A3, A3));
  q = fma2(t, q, make_float2(A2, A2));
  q = fma2(t, q, make_float2(A1, A1));
  const float2 w = mul2(mul2(t, q), g);
  return fma2(make_float2(-ax.x, -ax.y), w, make_float2(relu_nan(x.x), relu_nan(x.y)));
}

// Byte offsets of the regions of one CTA's dynamic shared memory.
struct SmemLayout {
  int ring;    // nslot * slot_bytes: weight slabs (with the unit's LayerNorm/bias vectors) streamed by the producer warp
  int ablk;    // [C][blk] f32: gathered residual columns, block c from CTA c; also the staging of outgoing partial sums
  int rs;      // [C][blk] f32: incoming partial sums of the second GEMM, block c from CTA c
  int xln;     // [Mp][lda] T: normalised rows, the first GEMM's A operand; aliased by the first GEMM's output
  int hblk;    // 2 x [C][M][npr] f32: the output head's gathered row partials by step parity (head_sep), else = ablk
  int hsrc;    // (2 or 1) x [M][npr] f32: this CTA's row partials for the head
  int pb;      // [M][PLD] f32: attention probabilities
  int oc;      // [Mp][ldo] T: attention output slice, A operand of the second GEMM
  int ac;      // [M][Ec] f32: this CTA's columns of the residual stream
  int acb;     // [M][Ec] bf16: copy of ac sent by the bf16 gather (operand type bf16)
  int cs;      // [3L][M][Ec] T: this CTA's columns of every unit's cache (or -1: caches in global memory)
  int kvs;     // [kv_slots][g][1+n_obs][kvw] f32: memory keys/values for cross-attention
  int cst;     // f32 constants: in_w[:, cols], in_b[cols], pos[:, cols], head_b, G, B (4-padded), gw[A][cols]
  int x;       // [M][A] f32: current sample x (replicated in every CTA of the cluster)
  int z;       // [M][A] f32: DDPM noise of the current step
  int sch;     // [T] u64: this job's lattice, bit b of word t = unit b refreshed at step t
  int stb;     // [T][8] f32: sampler coefficients of every step
  int psch;    // [T] u64: the producer warp's own copy of the job's refresh masks
  int bars;    // mbarriers: full[nslot], empty[nslot], cluster, xg, xr, xh
  int total;
};

struct JobParams {
  // model shape
  int L, E, nh, dh, H, A, n_obs, T, U, Cm;
  // decomposition
  int C, Ec, hid, g, M, Mp;
  int blk;                        // floats per exchange block (M*Ec + 4)
  int lda, ldg1, ldh, ldo, kvw;   // row strides (elements) of xln, q|k|v, hidden, attention output, memory k|v
  int lEc, lH;                    // log2 of Ec and H
  int n1[3];                      // first-GEMM width per unit kind (SA, CA, FFN)
  int hdr1[3];                    // header bytes of piece 1: first bias (LayerNorm shift folded in), second-GEMM bias slice
  int kv_slots;                   // L: memory keys/values of every layer prefetched per step; 1: per unit
  float invE;                     // 1 / E
  int kp_o, kp_h;                 // K of the second GEMMs (attention: Ec, FFN: hid), multiples of 16
  int n_jobs;
  int sampler, force;
  int nslot, slot_bytes;
  long long wait_limit;           // SM cycles before a wait gives up (WAIT_CYCLES_DEFAULT)
  int head_sep;                   // 1: head partials double-buffered by step parity; 0: one buffer + cluster barrier
  int npr;                        // floats per row of a head partial block: 2 + A, 4-padded
  // samples
  int samples;                    // real samples in this launch
  int per_sched;                  // samples that share one schedule
  int obs_mod;                    // obs / noise row of sample s = s % obs_mod
  // schedule lattice(s)
  const uint8_t* S;
  int S_rows;                     // 3L or L
  long long S_stride;             // bytes between schedules
  const int* sched_err;           // nonzero: schedule invalid, do nothing
  // sampler coefficients [T][8]
  const float* stab;
  // inputs / outputs
  const float* noise;             // [n_noise][obs_mod][H][A]
  const float* kv_obs;            // [obs_mod][n_obs][L][2E]
  const float* kv_time;           // [T][L][2E]
  float* out;                     // [samples][H][A]
  // packed weights: per CTA c, per layer: SA p1, SA p2, CA p1, CA p2, FFN p1, FFN p2
  const uint8_t* wpack;
  long long cta_stride, layer_stride;
  long long poff[3][2];           // piece byte offset within a layer block
  // float32 vectors
  const float* vec;
  long long v_inw, v_inb, v_pos, v_lnfg, v_lnfb, v_headw, v_headb;
  long long v_headG, v_headB;     // [A]: sum_e lnf_g[e] W_head[e][a], sum_e lnf_b[e] W_head[e][a]
  // caches [n_jobs][U][C][M][Ec] (dtype T), used when sm.cs < 0
  void* cache;
  float* trace;                   // [T][U][samples][H][E] or null
  int* status;
  SmemLayout sm;
};

// host helpers implemented in evo_job.cu
int  smem_layout(JobParams& p, int elem_bytes, int cache_smem);   // fills p.sm, returns total bytes
// compiled loop-kernel shapes (evo_shapes.h): id for a configuration or -1,
// with the ring geometry that shape was compiled for
int shape_find(int dtype, int E, int NH, int H, int C, int G, int* slot, int* nslot);
cudaError_t job_kernel_prepare(int shape, int smem_bytes, int* max_clusters);
cudaError_t launch_job(int shape, const JobParams& p, int n_clusters, cudaStream_t s);
// condition path; scratch holds 6E floats per token
cudaError_t launch_time_table(const float* wf32, const int* woff_dev, const int* woff, const float* kstep, int T,
                              int L, int E, float* scratch, float* kv_time, cudaStream_t s);
// condition path for at most 32 tokens of a bf16 model (cond_fast_ok): bf16 weight copy w16 =
// [E][4E] | [4E][E] | [E][L*2E] (row k holds every layer's [k | v] columns), bkv = [L*2E],
// part = cond_fast_part_floats floats, count = 768 zeroed counters (reset by the kernels)
bool cond_fast_ok(int E, int L, long long ntok);
size_t cond_fast_part_floats(int E, int L, long long ntok);
cudaError_t launch_obs_cond_fast(const float* wf32, const int* woff, const __nv_bfloat16* w16, const float* bkv,
                                 const float* obs, int N, int n_obs, int D, int L, int E, float* scratch,
                                 float* part, unsigned* count, float* kv_obs, cudaStream_t s);
cudaError_t launch_obs_cond(const float* wf32, const int* woff_dev, const int* woff, const float* obs, int N,
                            int n_obs, int D, int L, int E, float* scratch, float* kv_obs, cudaStream_t s);
cudaError_t launch_validate(const uint8_t* S, long long n, int* err, cudaStream_t s);
// one CTA, no cluster, no copies: waits on an mbarrier nothing arrives at through
// the loop kernel's helper (helper 0, limit in cycles) or the tensor-core
// kernels' helper (helper 1, limit in polls); the wait gives up and sets ST_TIMEOUT
cudaError_t launch_wait_probe(int helper, long long limit, int* status, cudaStream_t s);
cudaError_t launch_gelu_probe(const float* x, float* y, long long n, int packed, cudaStream_t s);
cudaError_t launch_pop_dev(const float* x, int P, int N_obs, int HA, float* dev, cudaStream_t s);

// batch-wide path (evo_wide.cu)
struct WideState;
struct WideCall {
  const float* obs;               // [obs_mod][n_obs][obs_dim]: the path computes kv_obs from these
  const float* noise;             // [n_noise][obs_mod][H][A]
  float* out;                     // [samples][H][A]: running x, final actions
  float* kv_obs;                  // [obs_mod][n_obs][L][2E] (output of the condition GEMMs)
  const float* kv_time;           // [T][L][2E]
  const float* stab;              // [T][8]
  int samples, per_sched, obs_mod;
  const uint8_t* S_host;          // [n_sched][S_rows][T], validated
  const uint8_t* S_dev;           // the same lattices on the device
  int n_sched, S_rows;
  float* trace;                   // [T][U][samples][H][E] or null: the residual added at every lattice cell
  int* status;
  cudaStream_t st;
};
bool wide_supported(const evo_config* c);
int wide_create(WideState** out, const evo_config* c, const float* weights, const float* wf32_dev, const int* woff,
                long long max_rows, int max_sched);   // evo_status
void wide_destroy(WideState* w);
long long wide_rows_capacity(const WideState* w);
const GuardList* wide_guards(const WideState* w);
long long wide_last_launches(const WideState* w);
cudaError_t wide_run(WideState* w, const WideCall& c);

// redundancy map and guided sampling (evo_redundancy.cu)
size_t redundancy_scratch_bytes(int T, int U, int N, int n, int metric);
bool redundancy_shape_ok(int T, int U, int N, int n, int metric);
cudaError_t launch_redundancy(const float* trace, int T, int U, int N, int n, int metric, float* d, void* scratch,
                              cudaStream_t st);
bool guided_shape_ok(int U, int T, int K, int gamma, int P);
cudaError_t launch_guided(const float* d, int U, int T, int K, float eps, int gamma, const uint64_t* rnd, int P,
                          uint8_t* S, cudaStream_t st);

// offsets (in floats) of the named tensors inside the float32 weight blob
enum WOff {
  W_OBS_W, W_OBS_B, W_COND_POS, W_CM_W1, W_CM_B1, W_CM_W2, W_CM_B2, W_IN_W, W_IN_B, W_POS,
  W_LAYER0,       // start of layer 0
  W_LAYER_STRIDE, // floats per layer
  // offsets inside one layer block
  WL_LN1G, WL_LN1B, WL_SA_WQKV, WL_SA_BQKV, WL_SA_WO, WL_SA_BO,
  WL_LN2G, WL_LN2B, WL_CA_WQ, WL_CA_BQ, WL_CA_WKV, WL_CA_BKV, WL_CA_WO, WL_CA_BO,
  WL_LN3G, WL_LN3B, WL_FF_W1, WL_FF_B1, WL_FF_W2, WL_FF_B2,
  W_LNF_G, W_LNF_B, W_HEAD_W, W_HEAD_B, W_TOTAL, W_COUNT
};

}  // namespace evo

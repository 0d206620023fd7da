// Internal declarations shared by the host API (evo_api.cu) and the kernels
// (evo_job.cu).  Not part of the C ABI.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

namespace evo {

constexpr int NCW = 8;              // compute warps per CTA
constexpr int NCT = NCW * 32;       // compute threads per CTA
constexpr int NTHREADS = NCT + 32;  // + one weight-streaming (producer) warp
constexpr int MAX_CLUSTER = 16;
constexpr int MAX_SLOTS = 8;

// error bits written to the device status word
constexpr int ST_SCHEDULE = 1;
constexpr int ST_TIMEOUT = 2;

// Byte offsets of the regions of one CTA's dynamic shared memory.
struct SmemLayout {
  int ring;    // nslot * slot_bytes, weight slabs streamed by the producer warp
  int afull;   // [Mp][ldf] f32: gathered residual rows; normalised in place into the GEMM A operand
  int hbuf;    // [M][ldf] f32: gathered rows for the output head (or -1: head uses afull)
  int rs;      // [C][M][Ec] f32: reduce-scatter landing zone of the second GEMM's partial sums
  int g1;      // first-GEMM output: q|k|v (f32, row stride ldg1) or FFN hidden (T, row stride ldh)
  int oc;      // [Mp][ldo] T: attention output slice, A operand of the second GEMM
  int ac;      // [M][Ec] f32: this CTA's columns of the residual stream
  int kvs;     // [g][1+n_obs][dh+Ec] f32: memory keys/values staged for one cross-attention unit
  int cst;     // in_w slice [A][Ec], in_b slice [Ec], pos slice [H][Ec] (f32)
  int x;       // [M][A] f32: current sample x (replicated in every CTA of the cluster)
  int z;       // [M][A] f32: DDPM noise of the current step
  int sch;     // [3L][T] u8: this job's lattice, one row per unit
  int bars;    // mbarriers: full[nslot], empty[nslot], cluster
  int total;
};

struct JobParams {
  // model shape
  int L, E, nh, dh, H, A, n_obs, T, U, Cm;
  // decomposition
  int C, Ec, hid, g, M, Mp;
  int ldf, ldg1, ldh, ldo;
  int n1_sa, n1_ca, n1_ff, n1max;
  int kp_o, kp_h;                 // padded K of the second GEMMs (attention: Ec, FFN: hid)
  int n_jobs;
  int sampler, force;
  int nslot, slot_bytes;
  int head_sep;
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
  long long v_ln, v_b1, v_b2, v_inw, v_inb, v_pos, v_lnfg, v_lnfb, v_headw, v_headb;
  // caches [n_jobs][U][C][M][Ec] (dtype T)
  void* cache;
  float* trace;                   // [T][U][samples][H][E] or null
  int* status;
  SmemLayout sm;
};

// host helpers implemented in evo_job.cu
int  smem_layout(JobParams& p, int elem_bytes);           // fills p.sm, returns total bytes
cudaError_t launch_job(const JobParams& p, int dtype, int n_clusters, cudaStream_t s);
cudaError_t job_kernel_prepare(int dtype, int smem_bytes, int cluster, int* max_clusters);
cudaError_t launch_time_table(const float* wf32, const int* woff, const float* stab_k, int T, int L, int E,
                              float* kv_time, cudaStream_t s);
cudaError_t launch_obs_cond(const float* wf32, const int* woff, const float* obs, int N, int n_obs, int D,
                            int L, int E, float* mem_scratch, float* kv_obs, cudaStream_t s);
cudaError_t launch_validate(const uint8_t* S, long long n, int* err, cudaStream_t s);
cudaError_t launch_pop_dev(const float* x, int P, int N_obs, int HA, float* dev, cudaStream_t s);

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

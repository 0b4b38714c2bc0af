// Device-side building blocks of the parallel decoder: grid barrier, embedding, LayerNorm
// prologue, batch-invariant skinny GEMM with fused epilogues (bias, activation, residual,
// K/V-cache scatter, LM-head argmax), attention over the key/value cache, and the
// fixed-point commit of the decoding algorithms.
//
// Batch invariance.  Every output element is produced by code whose arithmetic does not
// depend on how many rows a pass carries or on which slot a row sits in: a GEMM element is
// one warp's fixed-order dot product (each lane walks its K-chunks in order, then a fixed
// xor-butterfly); an attention row reduces over its keys in absolute key order; the argmax
// keeps the lowest index among equal maxima.  So a row's logits in a block pass are bit
// for bit those of the greedy pass at the same position whenever its inputs agree, which
// is what makes every parallel method return exactly the greedy tokens (Proposition 1).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "pd.h"

namespace pd {

constexpr int kThreads = 384;
constexpr int kWarps = kThreads / 32;
constexpr int kMTile = 8;           // rows per GEMM tile
constexpr int kNCol = 4;            // output columns per warp iteration (kNCol * kMTile == 32)
constexpr int kMaxLayers = 16;
constexpr int kMaxBatch = 64;        // sentences of one batched decode
constexpr int kMaxPassRows = 512;    // rows of one batched decoder pass
constexpr int kPageShift = 4;        // self-attention key/value cache pages of 16 positions
constexpr int kPageRows = 1 << kPageShift;
constexpr unsigned long long kWaitNs = 10000000000ull;  // bounded device waits: 10 s

enum Epi : int {
  EPI_STORE = 0,     // out = acc + bias
  EPI_ACT = 1,       // out_w = act(acc + bias), rounded to the weight type
  EPI_RESID = 2,     // out = acc + bias + resid
  EPI_QKV = 3,       // [q | k | v] = acc + bias -> q rows, k/v to cache slots
  EPI_KVCROSS = 4,   // columns of all decoder layers' [k | v] cross projections -> caches
  EPI_ARGMAX = 5,    // LM head: per-row running max / argmax / sum of exp
  EPI_LOGITS = 6     // LM head: store raw logits (test path)
};

template <typename W>
struct EncLayerW {
  const W *wqkv, *bqkv, *wo, *bo, *ln1g, *ln1b, *w1, *b1, *w2, *b2, *ln2g, *ln2b;
};
template <typename W>
struct DecLayerW {
  const W *wqkv, *bqkv, *wo, *bo, *ln1g, *ln1b, *wqc, *bqc, *wkvc, *bkvc, *woc, *boc, *ln2g,
      *ln2b, *w1, *b1, *w2, *b2, *ln3g, *ln3b;
};
template <typename W>
struct ModelW {
  const W* embed;
  const W* pos;
  const W *enc_lne_g, *enc_lne_b, *dec_lne_g, *dec_lne_b;
  const W *enc_lnf_g, *enc_lnf_b, *dec_lnf_g, *dec_lnf_b;
  EncLayerW<W> enc[kMaxLayers];
  DecLayerW<W> dec[kMaxLayers];
};

struct Dims {
  int d, H, dh, f, Le, Ld, V;
  int act, pre_ln, learned_pos, max_pos;
  int pad, eos, bos;
  float eps, emb_scale;
  int max_src, max_tgt;
  int max_keys;    // max(max_src, max_tgt): rows of the position table, keys of an attention row
  int max_batch;   // sentences one decode carries (cache slots per layer)
  int rows;        // activation rows: max(max_keys, min(max_batch * max_tgt, kMaxPassRows))
  int tc;          // bf16: GEMM phases on the tensor cores (else the SIMT path)
  int kv_pages;    // pages of kPageRows cache rows in each decoder layer's self K/V pool
  int pt_ld;       // page-table entries per sentence: ceil(max_tgt / kPageRows)
  int cl;          // cluster engine (cl_pass.cuh): decoder passes as per-layer super-phases
  int cl_n;        // cluster engine: clusters of the decode grid
  int cl_fu;       // cluster engine: FFN hidden units per CTA (cl_fu * kCl per cluster)
  int cl_np;       // cluster engine: partial sums a super-phase can leave (max(H, FFN slices))
};

// Per-CTA partial of the LM-head argmax for one row.
struct Partial {
  float mx;      // running max logit (-inf if the CTA saw no column)
  int idx;       // its lowest column index
  float sum;     // sum of exp(logit - mx) over the CTA's columns
  int nan;       // a NaN logit was seen
};

// Decoding state.  Every CTA keeps its own copy in shared memory and advances it by the same
// commit step from the same merged LM-head partials, so the copies stay identical; CTA 0
// writes the final one to device memory.
struct DecState {
  int method, b, max_len, h, stop_at_eos, max_passes, stop_rule;
  int b_eff, m_eff;       // current block size rule and system size (h for hybrid)
  int i, blk, k;          // block start (1-based), block length, passes in this block
  int ar_tail;            // hybrid: past h, one position per pass
  int n_iters, done, status, n_y, n_trace;
  int n_src;              // source length of the sentence (cross-attention keys)
  int scan;               // the first EOS of y_1..y_m is still to be found
  int a;                  // suffix rule: block positions i..i+a-1 already exact (not re-run)
  int init_rule;          // pd_init_rule: drafts of a new block
};

template <typename W>
struct Bufs {
  float *ra, *rb, *rc;         // residual-stream rows [rows][d]
  float *xa, *xb, *xc;         // normalised sublayer inputs (post-LN residuals) [rows][d]
  float *q, *k, *v;            // [rows][d]
  W* att;                      // [rows][d] attention output, rounded to W (the O input type)
  W* ffh;                      // [rows][f] FFN hidden, rounded to W (FFN2's input type)
  W *kself, *vself;            // [Ld][kv_pages * kPageRows][d]: pages of 16 positions, found
                               // through each sentence's page table
  W *kcross, *vcross;          // [Ld][max_batch * max_src][d]: sentence s at rows s * max_src..
  Partial* part;               // [grid][rows]
  DecState* st;
  pd_trace_step* trace;        // [max_tgt]
  int* trace_tok;              // [max_tgt][max_tgt]
  float* trace_prob;           // [max_tgt][max_tgt]
  unsigned* bar;               // [0] barrier counter, [1] abort flag
  int* src;                    // [max_src]
  int* dbg_tok;                // [max_tgt]
  float* pos_tab;              // sinusoidal positions [rows][d] (built once at create)
  int* page_tab;               // [max_batch][pt_ld] pool page of each sentence's 16-position
                               // page (written by the host before a decode)
  float* red;                  // bf16: split-K partial sums [S][rows][N]
  unsigned* cnt;               // bf16: split-K arrival counters (zero between uses)
  float* clp;                  // cluster engine: partial sums [2][cl_np][rows][d]
};

// ------------------------------------------------------------------------------------------
// small helpers
// ------------------------------------------------------------------------------------------

__device__ __forceinline__ unsigned long long globaltimer_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
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

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

// Weights are immutable while a kernel runs: read them through the non-coherent path.
__device__ __forceinline__ uint4 ldg_nc_v4(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ void unpack8(const uint4 u, float* f) {
  const unsigned w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}

__device__ __forceinline__ float act_fn(float v, int act) {
  if (act == PD_ACT_RELU) return fmaxf(v, 0.0f);
  if (act == PD_ACT_SILU) return v / (1.0f + expf(-v));
  return 0.5f * v * (1.0f + erff(v * 0.70710678118654752f));
}

// ------------------------------------------------------------------------------------------
// grid barriers with bounded waits
// ------------------------------------------------------------------------------------------



__device__ __forceinline__ void red_release_add(unsigned* p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Bar words: [0] arrival counter (only grows), [1] abort flag (words 2, 3 spare).  Spin until
// *word >= target; give up after kWaitNs, raising the abort flag
// and PD_ETIMEOUT, so that a broken schedule ends the kernel instead of hanging the GPU.
// The abort flag and the clock are looked at every 32nd poll only: a poll is then a single
// load, and the barrier is released one round trip after its last arrival.
__device__ __forceinline__ int spin_until(unsigned* bar, const unsigned* word, unsigned target,
                                          int* status,
                                          unsigned long long limit_ns = kWaitNs) {
  const unsigned long long t0 = globaltimer_ns();
  for (unsigned n = 1; ld_acquire_u32(word) < target; ++n) {
    if ((n & 31u) != 0u) continue;
    if (ld_acquire_u32(bar + 1) != 0u) return 0;
    if (globaltimer_ns() - t0 > limit_ns) {
      atomicExch(bar + 1, 1u);
      atomicCAS(status, 0, (int)PD_ETIMEOUT);
      return 0;
    }
  }
  return 1;
}

// Failure-detection check: one thread waits, with the barrier's bounded wait, for a counter
// that nothing advances (bar[0] stays 0, target 1).  The wait must give up after limit_ns,
// raise the abort flag and PD_ETIMEOUT in *status, and return.
__global__ void wait_probe_kernel(unsigned* bar, int* status, unsigned long long limit_ns) {
  if (blockIdx.x == 0 && threadIdx.x == 0) (void)spin_until(bar, bar, 1u, status, limit_ns);
}

// All CTAs of the (cooperatively launched, hence co-resident) grid meet here.  Release /
// acquire at GPU scope: the bar.sync before the release-add orders every thread's writes of
// this CTA before the arrival; the acquire load plus the bar.sync after it order the other
// CTAs' writes before every thread's later reads.  Returns false on abort.
// `during()` runs on every thread between this CTA's arrival and its wait (work that does not
// depend on the other CTAs, such as preparing the next phase).
template <typename F>
__device__ __forceinline__ bool grid_barrier(unsigned* bar, unsigned& target, int* status,
                                             F&& during) {
  __shared__ int s_ok;
  __syncthreads();
  target += gridDim.x;
  if (threadIdx.x == 0) {
    red_release_add(bar, 1u);
  }
  during();
  if (threadIdx.x == 0) {
    s_ok = spin_until(bar, bar, target, status);
  }
  __syncthreads();
  return s_ok != 0;
}
__device__ __forceinline__ bool grid_barrier(unsigned* bar, unsigned& target, int* status) {
  return grid_barrier(bar, target, status, [] {});
}

// Ask L2 to fetch [p, p + bytes) ahead of use (no data returns to the SM).  The weights of a
// phase do not depend on activations, so each CTA requests its own rows of the next phase
// before it waits at the barrier, overlapping the HBM latency with the wait.
__device__ __forceinline__ void l2_prefetch(const void* p, unsigned bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// Philox-4x32-10, the counter-based generator of Salmon, Moraes, Dror and Shaw ("Parallel
// random numbers: as easy as 1, 2, 3", SC 2011): ten rounds of two 32x32 -> 64-bit multiplies
// on a 4-word counter under a 2-word key bumped by the Weyl constants each round.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const unsigned long long p0 = 0xD2511F53ull * c.x, p1 = 0xCD9E8D57ull * c.z;
    const unsigned hi0 = (unsigned)(p0 >> 32), lo0 = (unsigned)p0;
    const unsigned hi1 = (unsigned)(p1 >> 32), lo1 = (unsigned)p1;
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
    k.x += 0x9E3779B9u;
    k.y += 0xBB67AE85u;
  }
  return c;
}

// Seeded weights of tensor number `tensor` of the blob (kind 0: std * z, z standard normal;
// 1: LayerNorm gain 1; 2: LayerNorm bias 0).  Element e draws Philox(counter (e / 2, tensor, 0,
// 0), key (seed, 0x5EED5EED)); its first two words u1, u2 (as (x + 0.5) / 2^32) give by
// Box-Muller z = sqrt(-2 ln u1) cos(2 pi u2) for even e, sin(2 pi u2) for odd e (in double
// precision), then std * z rounded to the weight type.
template <typename W>
__global__ void seeded_weights_kernel(W* dst, size_t n, unsigned tensor, unsigned seed, int kind,
                                      double std) {
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n;
       e += (size_t)gridDim.x * blockDim.x) {
    float v;
    if (kind == 1) {
      v = 1.0f;
    } else if (kind == 2) {
      v = 0.0f;
    } else {
      const uint4 r = philox4x32_10(make_uint4((unsigned)(e >> 1), tensor, 0u, 0u),
                                    make_uint2(seed, 0x5EED5EEDu));
      const double u1 = ((double)r.x + 0.5) * (1.0 / 4294967296.0);
      const double u2 = ((double)r.y + 0.5) * (1.0 / 4294967296.0);
      const double rad = sqrt(-2.0 * log(u1));
      const double ang = 6.283185307179586476925286766559 * u2;
      v = (float)(std * rad * ((e & 1) ? sin(ang) : cos(ang)));
    }
    dst[e] = from_f<W>(v);
  }
}

// Sinusoidal position table, row p = [sin(p w_k) | cos(p w_k)], w_k = 10000^(-2k/d), in double
// precision rounded to fp32 (run once when a context is created).
__global__ void sinusoid_kernel(float* tab, int rows, int d) {
  const int half = d / 2;
  for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < rows * d;
       idx += gridDim.x * blockDim.x) {
    const int p = idx / d, e = idx - p * d;
    const int k = e < half ? e : e - half;
    const double w = exp(-(2.0 * k / d) * log(10000.0));
    const double a = (double)p * w;
    tab[idx] = (float)(e < half ? sin(a) : cos(a));
  }
}

// ------------------------------------------------------------------------------------------
// GEMM phase: Y[M][N] = epilogue(X[M][K] . W[N][K]^T + bias), X = LN(x_src) or x_src
// ------------------------------------------------------------------------------------------

template <typename W>
struct GemmArgs {
  int M, N, K;
  // input rows X[M][K]: x_src rows, or (emb_tok != nullptr) the token embedding
  // E[tok] * sqrt(d) + position(pos0 + m); then optionally LayerNorm ln_a, the result stored
  // to x_store (fp32, by CTA 0), then optionally LayerNorm ln_b; X is rounded to W.
  const float* x_src;
  const W* xw_src;          // input rows already rounded to W (plain copy; instead of x_src)
  const int* emb_tok;
  const int* emb_pos;       // per-row positions of the embedded rows
  const W *ln_a_g, *ln_a_b;
  float* x_store;
  const W *ln_b_g, *ln_b_b;
  const W* w;               // [N][K]
  const W* bias;            // [N] or nullptr
  int epi;
  float* out;               // [M][ld] for STORE / RESID / LOGITS; q rows for QKV
  W* out_w;                 // [M][ld] for ACT
  int ld;
  const float* resid;       // [M][ld]
  W *kdst, *vdst;           // QKV: cache rows slot[m]; KVCROSS: cross caches
  float *kdst_f, *vdst_f;   // QKV into fp32 buffers (encoder)
  const int* slot;          // QKV into kdst / vdst: per-row cache slots
  Partial* part;            // ARGMAX: [grid][rows_ld]
  int part_ld;
  // How the phase is divided over the grid (gemm_plan): column groups, K-steps per warp,
  // warps per group, groups per CTA, groups per round; per warp its group slot and K part.
  int ngroups, spw, kw, gpc, stride;
  unsigned char wslot[kWarps], wpart[kWarps];
};

// Embedding and position tables (read by the GEMM whose input is the embedding).
template <typename W>
struct EmbedTabs {
  const W* E;               // token embedding [V][d]
  const W* P;               // learned positions [max_pos][d] (or nullptr)
  const float* ptab;        // sinusoidal positions [rows][d] (or nullptr)
};

// Reduce-scatter of 32 per-lane partial sums: afterwards lane L holds the warp total of value
// L.  Every value is summed over the lanes by the same balanced tree (pairs at lane distance
// 16, 8, 4, 2, 1), so the result of a value does not depend on its index.
__device__ __forceinline__ float reduce_scatter32(float (&v)[32]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int s = 16; s >= 1; s >>= 1) {
    const bool upper = (lane & s) != 0;
#pragma unroll
    for (int j = 0; j < s; ++j) {
      const float send = upper ? v[j] : v[j + s];
      const float keep = upper ? v[j + s] : v[j];
      v[j] = keep + __shfl_xor_sync(0xffffffffu, send, s);
    }
  }
  return v[0];
}

// Elements one warp covers per 16-byte load of every lane (one "K-step").
template <typename W> struct KStep { static constexpr int E = 32 * 16 / (int)sizeof(W); };

// Partial dot products of kNCol output columns n0.. for up to kMTile rows over the K-steps
// s0..s0+ns-1 (ns <= 2): all weight loads of the warp are issued before the first FMA, each
// element is accumulated in ascending K order, then the reduce-scatter leaves value
// (column c, row r) on lane c * kMTile + r.
__device__ __forceinline__ float dot_part(const __nv_bfloat16* __restrict__ w, int K, int n0,
                                          int nvalid, const __nv_bfloat16* xs, int mt, int s0,
                                          int ns) {
  const int lane = threadIdx.x & 31;
  uint4 wr[2][kNCol];
#pragma unroll
  for (int t = 0; t < 2; ++t)
#pragma unroll
    for (int c = 0; c < kNCol; ++c)
      wr[t][c] = (t < ns && c < nvalid)
                     ? ldg_nc_v4(w + (size_t)(n0 + c) * K + (s0 + t) * 256 + lane * 8)
                     : make_uint4(0u, 0u, 0u, 0u);
  float acc[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) acc[i] = 0.f;
#pragma unroll
  for (int t = 0; t < 2; ++t) {
    if (t < ns) {
      float wv[kNCol][8];
#pragma unroll
      for (int c = 0; c < kNCol; ++c) unpack8(wr[t][c], wv[c]);
#pragma unroll
      for (int r = 0; r < kMTile; ++r) {
        if (r < mt) {
          float x[8];
          unpack8(*reinterpret_cast<const uint4*>(xs + (size_t)r * K + (s0 + t) * 256 + lane * 8), x);
#pragma unroll
          for (int c = 0; c < kNCol; ++c)
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[c * kMTile + r] = fmaf(wv[c][e], x[e], acc[c * kMTile + r]);
        }
      }
    }
  }
  return reduce_scatter32(acc);
}

__device__ __forceinline__ float dot_part(const float* __restrict__ w, int K, int n0, int nvalid,
                                          const float* xs, int mt, int s0, int ns) {
  const int lane = threadIdx.x & 31;
  uint4 wr[2][kNCol];
#pragma unroll
  for (int t = 0; t < 2; ++t)
#pragma unroll
    for (int c = 0; c < kNCol; ++c)
      wr[t][c] = (t < ns && c < nvalid)
                     ? ldg_nc_v4(w + (size_t)(n0 + c) * K + (s0 + t) * 128 + lane * 4)
                     : make_uint4(0u, 0u, 0u, 0u);
  float acc[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) acc[i] = 0.f;
#pragma unroll
  for (int t = 0; t < 2; ++t) {
    if (t < ns) {
#pragma unroll
      for (int r = 0; r < kMTile; ++r) {
        if (r < mt) {
          const float4 x =
              *reinterpret_cast<const float4*>(xs + (size_t)r * K + (s0 + t) * 128 + lane * 4);
#pragma unroll
          for (int c = 0; c < kNCol; ++c) {
            float& a = acc[c * kMTile + r];
            a = fmaf(__uint_as_float(wr[t][c].x), x.x, a);
            a = fmaf(__uint_as_float(wr[t][c].y), x.y, a);
            a = fmaf(__uint_as_float(wr[t][c].z), x.z, a);
            a = fmaf(__uint_as_float(wr[t][c].w), x.w, a);
          }
        }
      }
    }
  }
  return reduce_scatter32(acc);
}

constexpr int kMaxRowRegs = 8;      // embedded / normalised rows: <= 8 float4 per lane
constexpr int kStageB = 4;
__device__ __forceinline__ uint4 ld_act16(const void* p) {
  uint4 v;
  asm volatile("ld.global.cg.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Four consecutive elements p[0..3] as floats, one vector load (p is 4-element aligned: every
// tensor of the weight blob and every shared-memory copy starts at a multiple of 256 elements).
__device__ __forceinline__ float4 get4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ float4 get4(const __nv_bfloat16* p) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);      // bf16 = the high half of a float
  return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                     __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
}

// LayerNorm of a row held as float4 v[i] = elements lane*4 + 128*i: mean and biased variance
// from per-lane sums in ascending i, then fixed butterflies.
template <typename W>
__device__ __forceinline__ void ln_regs(float4 (&v)[kMaxRowRegs], int nI, int K, const W* g,
                                        const W* b, float eps) {
  const int lane = threadIdx.x & 31;
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < kMaxRowRegs; ++i)
    if (i < nI) s += (v[i].x + v[i].y) + (v[i].z + v[i].w);
  const float mean = warp_sum(s) / K;
  float s2 = 0.f;
#pragma unroll
  for (int i = 0; i < kMaxRowRegs; ++i) {
    if (i < nI) {
      const float a = v[i].x - mean, bb = v[i].y - mean, c = v[i].z - mean, d = v[i].w - mean;
      s2 += (a * a + bb * bb) + (c * c + d * d);
    }
  }
  const float rstd = 1.0f / sqrtf(warp_sum(s2) / K + eps);
#pragma unroll
  for (int i = 0; i < kMaxRowRegs; ++i) {
    if (i < nI) {
      const int k = lane * 4 + 128 * i;
      const float4 gk = get4(g + k), bk = get4(b + k);
      v[i].x = (v[i].x - mean) * rstd * gk.x + bk.x;
      v[i].y = (v[i].y - mean) * rstd * gk.y + bk.y;
      v[i].z = (v[i].z - mean) * rstd * gk.z + bk.z;
      v[i].w = (v[i].w - mean) * rstd * gk.w + bk.w;
    }
  }
}

__device__ __forceinline__ void put4(float* xs, float4 v) { *reinterpret_cast<float4*>(xs) = v; }
__device__ __forceinline__ void put4(__nv_bfloat16* xs, float4 v) {
  __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
  uint2 u;
  u.x = *reinterpret_cast<unsigned*>(&a);
  u.y = *reinterpret_cast<unsigned*>(&b);
  *reinterpret_cast<uint2*>(xs) = u;
}


// Stage rows m0..m0+mt of the GEMM input into shared memory (one warp per row, each element
// loaded once into registers).
template <typename W>
__device__ void stage_x(const GemmArgs<W>& g, const EmbedTabs<W>& T, const Dims& D, int m0,
                        int mt, W* xs) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int K = g.K;
  const bool any_ln = g.ln_a_g != nullptr || g.ln_b_g != nullptr || g.emb_tok != nullptr;
  if (!any_ln) {
    // plain copy, all threads, 16-byte items: fp32 rows (4 elements, rounded to W, optionally
    // stored to x_store) or rows already in W (16 / sizeof(W) elements, copied as they are)
    const bool wsrc = g.xw_src != nullptr;
    const bool store = g.x_store != nullptr && blockIdx.x == 0;
    const int E = wsrc ? 16 / (int)sizeof(W) : 4;
    const int es = wsrc ? (int)sizeof(W) : 4;
    const char* src = wsrc ? reinterpret_cast<const char*>(g.xw_src)
                           : reinterpret_cast<const char*>(g.x_src);
    const int KE = K / E, F = mt * KE;
    for (int f0 = 0; f0 < F; f0 += kThreads * kStageB) {
      uint4 v[kStageB];
#pragma unroll
      for (int j = 0; j < kStageB; ++j) {
        const int f = f0 + j * kThreads + (int)threadIdx.x;
        if (f < F) {
          const int r = f / KE, k = (f - r * KE) * E;
          v[j] = ld_act16(src + ((size_t)(m0 + r) * K + k) * es);
        }
      }
#pragma unroll
      for (int j = 0; j < kStageB; ++j) {
        const int f = f0 + j * kThreads + (int)threadIdx.x;
        if (f < F) {
          const int r = f / KE, k = (f - r * KE) * E;
          if (wsrc) {
            *reinterpret_cast<uint4*>(xs + (size_t)r * K + k) = v[j];
          } else {
            const float4 x = make_float4(__uint_as_float(v[j].x), __uint_as_float(v[j].y),
                                         __uint_as_float(v[j].z), __uint_as_float(v[j].w));
            if (store) *reinterpret_cast<float4*>(g.x_store + (size_t)(m0 + r) * K + k) = x;
            put4(xs + (size_t)r * K + k, x);
          }
        }
      }
    }
    return;
  }
  for (int r = warp; r < mt; r += kWarps) {
    const int m = m0 + r;
    const bool store = g.x_store != nullptr && blockIdx.x == 0;
    const int nI = K / 128;              // K <= 1024 for rows that are embedded or normalised
    float4 v[kMaxRowRegs];
    if (g.emb_tok != nullptr) {
      int t = g.emb_tok[m];
      t = t < 0 ? 0 : (t >= D.V ? D.V - 1 : t);
      const int p = g.emb_pos[m];
      const W* er = T.E + (size_t)t * K;
#pragma unroll
      for (int i = 0; i < kMaxRowRegs; ++i) {
        if (i < nI) {
          const int k = lane * 4 + 128 * i;
          const float4 e = get4(er + k);
          float4 ps;
          if (T.P != nullptr) ps = get4(T.P + (size_t)(p < D.max_pos ? p : D.max_pos - 1) * K + k);
          else ps = *reinterpret_cast<const float4*>(T.ptab + (size_t)p * K + k);
          v[i] = make_float4(e.x * D.emb_scale + ps.x, e.y * D.emb_scale + ps.y,
                             e.z * D.emb_scale + ps.z, e.w * D.emb_scale + ps.w);
        }
      }
    } else {
      const float* src = g.x_src + (size_t)m * K;
#pragma unroll
      for (int i = 0; i < kMaxRowRegs; ++i)
        if (i < nI) v[i] = *reinterpret_cast<const float4*>(src + lane * 4 + 128 * i);
    }
    if (g.ln_a_g != nullptr) ln_regs(v, nI, K, g.ln_a_g, g.ln_a_b, D.eps);
    if (store) {
#pragma unroll
      for (int i = 0; i < kMaxRowRegs; ++i)
        if (i < nI)
          *reinterpret_cast<float4*>(g.x_store + (size_t)m * K + lane * 4 + 128 * i) = v[i];
    }
    if (g.ln_b_g != nullptr) ln_regs(v, nI, K, g.ln_b_g, g.ln_b_b, D.eps);
#pragma unroll
    for (int i = 0; i < kMaxRowRegs; ++i)
      if (i < nI) put4(xs + (size_t)r * K + lane * 4 + 128 * i, v[i]);
  }
}

// Bulk L2 prefetch of the weight rows this CTA's warps will read in a GEMM phase over N
// columns of K (the same column groups gemm_phase assigns them).
template <typename W>
__device__ __forceinline__ void prefetch_gemm_weights(const W* w, int N, int K) {
  if (w == nullptr) return;
  const int ngroups = (N + kNCol - 1) / kNCol;
  for (int gi = blockIdx.x + (int)(threadIdx.x >> 5) * gridDim.x; gi < ngroups;
       gi += gridDim.x * kWarps) {
    if ((threadIdx.x & 31) != 0) continue;
    const int n0 = gi * kNCol;
    const int nv = N - n0 < kNCol ? N - n0 : kNCol;
    l2_prefetch(w + (size_t)n0 * K, (unsigned)(nv * K * sizeof(W)));
  }
}

__device__ __forceinline__ void argmax_push(float v, int col, float& mx, int& idx, float& sum,
                                            int& nan) {
  if (v != v) { nan = 1; return; }
  if (v > mx) {
    sum = (mx == -INFINITY ? 0.f : sum * expf(mx - v)) + 1.0f;
    mx = v;
    idx = col;
  } else {
    sum += expf(v - mx);
    if (v == mx && col < idx) idx = col;
  }
}

__device__ __forceinline__ Partial shfl_partial(const Partial& a, int o) {
  Partial b;
  b.mx = __shfl_xor_sync(0xffffffffu, a.mx, o);
  b.idx = __shfl_xor_sync(0xffffffffu, a.idx, o);
  b.sum = __shfl_xor_sync(0xffffffffu, a.sum, o);
  b.nan = __shfl_xor_sync(0xffffffffu, a.nan, o);
  return b;
}

// a <- a (+) b: larger max wins, equal maxima keep the lower index; sums rescaled.
__device__ __forceinline__ void partial_merge(Partial& a, const Partial& b) {
  a.nan |= b.nan;
  if (b.mx == -INFINITY) return;
  if (a.mx == -INFINITY) { a.mx = b.mx; a.idx = b.idx; a.sum = b.sum; return; }
  if (b.mx > a.mx) {
    a.sum = a.sum * expf(a.mx - b.mx) + b.sum;
    a.mx = b.mx;
    a.idx = b.idx;
  } else {
    a.sum = a.sum + b.sum * expf(b.mx - a.mx);
    if (b.mx == a.mx && b.idx < a.idx) a.idx = b.idx;
  }
}

// The division of a GEMM phase over the grid, a function of N, K and the grid only: K-steps
// per warp are 1 when the phase then still fits in one round over the grid (shorter dot chains
// for the small GEMMs), else 2.  Computed once per phase by the thread that writes the
// arguments, off the phase's chain of dependent steps.
template <typename W>
__device__ __forceinline__ void gemm_plan(GemmArgs<W>& g, int grid) {
  const int steps = g.K / KStep<W>::E;
  g.ngroups = (g.N + kNCol - 1) / kNCol;
  g.spw = (steps <= kWarps && g.ngroups <= grid * (kWarps / steps)) ? 1 : 2;
  g.kw = (steps + g.spw - 1) / g.spw;
  g.gpc = kWarps / g.kw;
  g.stride = grid * g.gpc;
  for (int w = 0, sl = 0, pt = 0; w < kWarps; ++w) {
    g.wslot[w] = (unsigned char)sl;
    g.wpart[w] = (unsigned char)pt;
    if (++pt == g.kw) { pt = 0; ++sl; }
  }
}

// GEMM phase.  N is cut into column groups of kNCol; a group is computed by kw warps of one
// CTA, warp j covering K-steps 2j and 2j+1 (kw = ceil(K-steps / 2), a function of K only),
// and their partial sums are added in warp order.  Groups are dealt to CTAs round robin
// (group g -> CTA g mod grid), so that even a 512-column phase spreads over 128 SMs.
template <typename W>
__device__ __noinline__ void gemm_phase(const GemmArgs<W>& g, const EmbedTabs<W>& T,
                                        const Dims& D, unsigned char* smem) {
  W* xs = reinterpret_cast<W*>(smem);
  unsigned char* small = smem + (size_t)kMTile * (D.d > D.f ? D.d : D.f) * sizeof(W);
  Partial* ps = reinterpret_cast<Partial*>(small);        // [kWarps][32]
  float* red = reinterpret_cast<float*>(small);           // [kWarps][32] (not used with ps)
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int steps = g.K / KStep<W>::E;
  const int ngroups = g.ngroups, spw = g.spw, kw = g.kw, gpc = g.gpc, stride = g.stride;
  const int slot = g.wslot[warp], part = g.wpart[warp];
  const int s0 = spw * part, ns = steps - s0 < spw ? steps - s0 : spw;
  const int c = lane / kMTile, r = lane % kMTile;   // the (column, row) this lane finishes
  for (int m0 = 0; m0 < g.M; m0 += kMTile) {
    const int mt = g.M - m0 < kMTile ? g.M - m0 : kMTile;
    __syncthreads();
    stage_x(g, T, D, m0, mt, xs);
    __syncthreads();
    float amx = -INFINITY, asum = 0.f;
    int aidx = 0x7fffffff, anan = 0;
    for (int base = 0; base < ngroups; base += stride) {
      const int gi = base + slot * gridDim.x + blockIdx.x;
      const bool active = slot < gpc && gi < ngroups;
      const int n0 = gi * kNCol;
      const int nvalid = active ? (g.N - n0 < kNCol ? g.N - n0 : kNCol) : 0;
      float a = 0.f;
      if (active) a = dot_part(g.w, g.K, n0, nvalid, xs, mt, s0, ns);
      if (kw > 1) {
        if (active) red[warp * 32 + lane] = a;
        __syncthreads();
        if (active && part == 0)
          for (int j = 1; j < kw; ++j) a += red[(warp + j) * 32 + lane];
        __syncthreads();
      }
      if (!active || part != 0 || r >= mt || c >= nvalid) continue;
      const int m = m0 + r, n = n0 + c;
      const float bias = g.bias != nullptr ? to_f(g.bias[n]) : 0.f;
      const float v = a + bias;
      switch (g.epi) {
        case EPI_STORE: g.out[(size_t)m * g.ld + n] = v; break;
        case EPI_ACT: g.out_w[(size_t)m * g.ld + n] = from_f<W>(act_fn(v, D.act)); break;
        case EPI_RESID: g.out[(size_t)m * g.ld + n] = v + g.resid[(size_t)m * g.ld + n]; break;
        case EPI_QKV: {
          const int which = n / D.d, cc = n - which * D.d;
          if (which == 0) {
            g.out[(size_t)m * D.d + cc] = v;
          } else if (g.kdst != nullptr) {
            W* dst = which == 1 ? g.kdst : g.vdst;
            dst[(size_t)g.slot[m] * D.d + cc] = from_f<W>(v);
          } else {
            float* dst = which == 1 ? g.kdst_f : g.vdst_f;
            dst[(size_t)m * D.d + cc] = v;
          }
          break;
        }
        case EPI_KVCROSS: {
          const int which = n / D.d, cc = n - which * D.d;
          W* dst = which == 0 ? g.kdst : g.vdst;
          dst[(size_t)m * D.d + cc] = from_f<W>(v);
          break;
        }
        case EPI_ARGMAX: argmax_push(v, n, amx, aidx, asum, anan); break;
        case EPI_LOGITS: g.out[(size_t)m * g.ld + n] = v; break;
      }
    }
    if (g.epi == EPI_ARGMAX) {
      // lane c*kMTile + r of a part-0 warp holds row r over its columns n0 + c.  Row r's
      // kWarps * kNCol partials are merged by warp r: lane l takes entries l, l + 32, ...
      // (entry e = warp w2, column c2 with e = w2 * kNCol + c2), then a fixed butterfly; the
      // CTA partial of the row is published
      __syncthreads();
      ps[warp * 32 + lane] = Partial{amx, aidx, asum, anan};
      __syncthreads();
      for (int rr = warp; rr < mt; rr += kWarps) {
        Partial acc{-INFINITY, 0x7fffffff, 0.f, 0};
        for (int e = lane; e < kWarps * kNCol; e += 32)
          partial_merge(acc, ps[(e / kNCol) * 32 + (e % kNCol) * kMTile + rr]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) partial_merge(acc, shfl_partial(acc, o));
        if (lane == 0) g.part[(size_t)blockIdx.x * g.part_ld + m0 + rr] = acc;
      }
    }
  }
}

// ------------------------------------------------------------------------------------------
// attention: out[m, head] = softmax(q k^T / sqrt(dh)) v over keys 0..T(m)-1, stored as O
// ------------------------------------------------------------------------------------------

template <typename KV>
__device__ __forceinline__ float key_dot(const KV* krow, const float* qs, int dh);

template <>
__device__ __forceinline__ float key_dot<__nv_bfloat16>(const __nv_bfloat16* krow,
                                                        const float* qs, int dh) {
  float s = 0.f;
  for (int e = 0; e < dh; e += 8) {
    float k[8];
    unpack8(*reinterpret_cast<const uint4*>(krow + e), k);
#pragma unroll
    for (int t = 0; t < 8; ++t) s = fmaf(qs[e + t], k[t], s);
  }
  return s;
}

template <>
__device__ __forceinline__ float key_dot<float>(const float* krow, const float* qs, int dh) {
  float s = 0.f;
  for (int e = 0; e < dh; e += 4) {
    const float4 k = *reinterpret_cast<const float4*>(krow + e);
    s = fmaf(qs[e], k.x, s);
    s = fmaf(qs[e + 1], k.y, s);
    s = fmaf(qs[e + 2], k.z, s);
    s = fmaf(qs[e + 3], k.w, s);
  }
  return s;
}

// acc[e] += p * v[e] for 32 consecutive value elements of one key.
__device__ __forceinline__ void add_pv32(const __nv_bfloat16* v, float p, float (&acc)[32]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float f[8];
    unpack8(*reinterpret_cast<const uint4*>(v + 8 * i), f);
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[8 * i + e] = fmaf(p, f[e], acc[8 * i + e]);
  }
}
__device__ __forceinline__ void add_pv32(const float* v, float p, float (&acc)[32]) {
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float4 f = *reinterpret_cast<const float4*>(v + 4 * i);
    acc[4 * i] = fmaf(p, f.x, acc[4 * i]);
    acc[4 * i + 1] = fmaf(p, f.y, acc[4 * i + 1]);
    acc[4 * i + 2] = fmaf(p, f.z, acc[4 * i + 2]);
    acc[4 * i + 3] = fmaf(p, f.w, acc[4 * i + 3]);
  }
}

// One warp per (row m, head): lane l owns keys l, l+32, ...  Scores, softmax and the
// p-weighted value sums are accumulated per lane in ascending key order, then combined by
// fixed butterflies, so a row's result depends only on its own query and keys.
// Row m attends rkeys[m] keys of kc / vc (causal rows pass their position + 1); without the
// arrays every row attends the first n_keys keys.  Key j of row m is at key row rbase[m] + j
// (contiguous caches), or, given a page table ptab ([sentence][pt_ld], the paged self-attention
// cache), rbase[m] is the row's sentence s and key j sits in pool page ptab[s][j / 16] at
// row j % 16.
template <typename KV>
__device__ __forceinline__ size_t key_row(const int* ptab, int pt_ld, int base, int j) {
  return ptab != nullptr
             ? (size_t)ptab[base * pt_ld + (j >> kPageShift)] * kPageRows + (j & (kPageRows - 1))
             : (size_t)base + j;
}
template <typename KV, typename O>
__device__ __noinline__ void attn_phase(const Dims& D, const float* q, const KV* kc, const KV* vc,
                           O* out, int M, const int* rbase, const int* rkeys, int n_keys,
                           float* scratch, const int* ptab = nullptr) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int gw = warp * gridDim.x + blockIdx.x;     // items dealt to CTAs round robin
  const int tw = gridDim.x * kWarps;
  const int dh = D.dh;
  float* qs = scratch + (size_t)warp * (128 + D.max_keys + 4);
  float* ps = qs + 128;
  const float scale = 1.0f / sqrtf((float)dh);
  for (int it = gw; it < M * D.H; it += tw) {
    const int m = it / D.H, h = it - m * D.H;
    const int T = rkeys != nullptr ? rkeys[m] : n_keys;
    const int base = rbase != nullptr ? rbase[m] : 0;
    for (int e = lane; e < dh; e += 32) qs[e] = q[(size_t)m * D.d + h * dh + e] * scale;
    __syncwarp();
    float lmax = -INFINITY;
    for (int j = lane; j < T; j += 32) {
      const float s = key_dot<KV>(kc + key_row<KV>(ptab, D.pt_ld, base, j) * D.d + h * dh, qs, dh);
      ps[j] = s;
      lmax = fmaxf(lmax, s);
    }
    const float mx = warp_max(lmax);
    float lsum = 0.f;
    for (int j = lane; j < T; j += 32) {
      const float p = expf(ps[j] - mx);
      ps[j] = p;
      lsum += p;
    }
    const float sum = warp_sum(lsum);
    for (int c0 = 0; c0 < dh; c0 += 32) {
      float acc[32];
#pragma unroll
      for (int e = 0; e < 32; ++e) acc[e] = 0.f;
      for (int j = lane; j < T; j += 32) {
        const float p = ps[j];
        add_pv32(vc + key_row<KV>(ptab, D.pt_ld, base, j) * D.d + h * dh + c0, p, acc);
      }
      const float tot = reduce_scatter32(acc);
      out[(size_t)m * D.d + h * dh + c0 + lane] = from_f<O>(tot / sum);
    }
    __syncwarp();
  }
}

}  // namespace pd

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

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kMTile = 16;          // rows per GEMM tile
constexpr int kMaxLayers = 16;
constexpr unsigned long long kWaitNs = 10000000000ull;  // bounded device waits: 10 s

enum Epi : int {
  EPI_STORE = 0,     // out = acc + bias
  EPI_ACT = 1,       // out = act(acc + bias)
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
  int max_src, max_tgt, rows;   // rows = max(max_src, max_tgt): activation buffer rows
};

// Per-CTA partial of the LM-head argmax for one row.
struct Partial {
  float mx;      // running max logit (-inf if the CTA saw no column)
  int idx;       // its lowest column index
  float sum;     // sum of exp(logit - mx) over the CTA's columns
  int nan;       // a NaN logit was seen
};

// Decoding state, in device memory, advanced by the commit step.
struct DecState {
  int method, b, max_len, h, stop_at_eos, max_passes;
  int b_eff, m_eff;       // current block size rule and system size (h for hybrid)
  int i, blk, k;          // block start (1-based), block length, passes in this block
  int ar_tail;            // hybrid: past h, one position per pass
  int n_iters, done, status, n_y, n_trace;
};

template <typename W>
struct Bufs {
  float *ra, *rb, *rc;         // residual-stream rows [rows][d]
  float *xa, *xb, *xc;         // normalised sublayer inputs (post-LN residuals) [rows][d]
  float *q, *k, *v, *att;      // [rows][d]
  float* ffh;                  // [rows][f]
  W *kself, *vself;            // [Ld][max_tgt][d]
  W *kcross, *vcross;          // [Ld][max_src][d]
  Partial* part;               // [grid][rows]
  int* y;                      // [max_tgt + 1]: y_0 = BOS, then the draft / solution
  DecState* st;
  pd_trace_step* trace;        // [max_tgt]
  int* trace_tok;              // [max_tgt][max_tgt]
  float* trace_prob;           // [max_tgt][max_tgt]
  unsigned* bar;               // [0] barrier counter, [1] abort flag
  int* src;                    // [max_src]
  int* dbg_tok;                // [max_tgt]
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
// grid barrier with a bounded wait
// ------------------------------------------------------------------------------------------

// All CTAs of the (cooperatively launched, hence co-resident) grid meet here.  The counter
// only grows; `target` tracks how far it must have grown.  A CTA that waits longer than
// kWaitNs raises the abort flag and records PD_ETIMEOUT; every CTA leaves on abort, so a
// broken schedule ends the kernel instead of hanging the GPU.  Returns false on abort.
__device__ __forceinline__ bool grid_barrier(unsigned* bar, unsigned& target, int* status) {
  __shared__ int s_ok;
  __syncthreads();
  target += gridDim.x;
  if (threadIdx.x == 0) {
    __threadfence();
    atomicAdd(bar, 1u);
    int ok = 1;
    const unsigned long long t0 = globaltimer_ns();
    while (ld_acquire_u32(bar) < target) {
      if (ld_acquire_u32(bar + 1) != 0u) { ok = 0; break; }
      if (globaltimer_ns() - t0 > kWaitNs) {
        atomicExch(bar + 1, 1u);
        atomicCAS(status, 0, (int)PD_ETIMEOUT);
        ok = 0;
        break;
      }
    }
    __threadfence();
    s_ok = ok;
  }
  __syncthreads();
  return s_ok != 0;
}

// ------------------------------------------------------------------------------------------
// embedding: x = E[tok] * sqrt(d) + pos(p)  (+ embedding LayerNorm for pre-LN models)
// ------------------------------------------------------------------------------------------

template <typename W>
__device__ void embed_phase(const Dims& D, const W* __restrict__ E, const W* __restrict__ P,
                            const W* lng, const W* lnb, const int* tok, int pos0, int M,
                            float* out) {
  const int lane = threadIdx.x & 31;
  const int gw = blockIdx.x * kWarps + (threadIdx.x >> 5);
  const int tw = gridDim.x * kWarps;
  for (int m = gw; m < M; m += tw) {
    int t = __ldcg(tok + m);
    t = t < 0 ? 0 : (t >= D.V ? D.V - 1 : t);
    const int p = pos0 + m;
    float* o = out + (size_t)m * D.d;
    const int half = D.d / 2;
    for (int e = lane; e < D.d; e += 32) {
      float v = to_f(E[(size_t)t * D.d + e]) * D.emb_scale;
      if (D.learned_pos) {
        v += to_f(P[(size_t)(p < D.max_pos ? p : D.max_pos - 1) * D.d + e]);
      } else {
        const int kk = e < half ? e : e - half;
        const double w = exp(-(2.0 * kk / D.d) * log(10000.0));
        const double a = (double)p * w;
        v += (float)(e < half ? sin(a) : cos(a));
      }
      o[e] = v;
    }
    if (lng != nullptr) {
      __syncwarp();
      float s = 0.f;
      for (int e = lane; e < D.d; e += 32) s += o[e];
      const float mean = warp_sum(s) / D.d;
      float s2 = 0.f;
      for (int e = lane; e < D.d; e += 32) { const float c = o[e] - mean; s2 += c * c; }
      const float rstd = 1.0f / sqrtf(warp_sum(s2) / D.d + D.eps);
      for (int e = lane; e < D.d; e += 32)
        o[e] = (o[e] - mean) * rstd * to_f(lng[e]) + to_f(lnb[e]);
    }
  }
}

// ------------------------------------------------------------------------------------------
// GEMM phase: Y[M][N] = epilogue(X[M][K] . W[N][K]^T + bias), X = LN(x_src) or x_src
// ------------------------------------------------------------------------------------------

template <typename W>
struct GemmArgs {
  int M, N, K;
  const float* x_src;       // [M][K] fp32 rows
  const W *x_g, *x_b;       // LayerNorm of the input rows (nullptr: none)
  float* x_store;           // write the normalised fp32 input rows here (nullptr: no)
  const W* w;               // [N][K]
  const W* bias;            // [N] or nullptr
  int epi;
  float* out;               // [M][ld] for STORE / ACT / RESID / LOGITS; q rows for QKV
  int ld;
  const float* resid;       // [M][ld]
  W *kdst, *vdst;           // QKV: cache rows (slot = slot0 + m); KVCROSS: cross caches
  float *kdst_f, *vdst_f;   // QKV into fp32 buffers (encoder)
  int slot0;
  int kv_ld;                // KVCROSS: rows per layer in the cross cache (max_src)
  Partial* part;            // ARGMAX: [grid][rows_ld]
  int part_ld;
};

// One output column for up to kMTile rows: each lane walks its K-chunks in ascending order,
// then a fixed xor-butterfly; every lane ends with the same sums.
__device__ __forceinline__ void dot_col(const __nv_bfloat16* __restrict__ wrow,
                                        const __nv_bfloat16* xs, int K, int mt,
                                        float (&acc)[kMTile]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int r = 0; r < kMTile; ++r) acc[r] = 0.f;
#pragma unroll 2
  for (int k0 = lane * 8; k0 < K; k0 += 256) {
    float w[8];
    unpack8(ldg_nc_v4(wrow + k0), w);
#pragma unroll
    for (int r = 0; r < kMTile; ++r) {
      if (r < mt) {
        float x[8];
        unpack8(*reinterpret_cast<const uint4*>(xs + (size_t)r * K + k0), x);
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[r] = fmaf(w[e], x[e], acc[r]);
      }
    }
  }
#pragma unroll
  for (int r = 0; r < kMTile; ++r) acc[r] = warp_sum(acc[r]);
}

__device__ __forceinline__ void dot_col(const float* __restrict__ wrow, const float* xs, int K,
                                        int mt, float (&acc)[kMTile]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int r = 0; r < kMTile; ++r) acc[r] = 0.f;
#pragma unroll 2
  for (int k0 = lane * 4; k0 < K; k0 += 128) {
    const uint4 wu = ldg_nc_v4(wrow + k0);
    const float w[4] = {__uint_as_float(wu.x), __uint_as_float(wu.y), __uint_as_float(wu.z),
                        __uint_as_float(wu.w)};
#pragma unroll
    for (int r = 0; r < kMTile; ++r) {
      if (r < mt) {
        const float4 x = *reinterpret_cast<const float4*>(xs + (size_t)r * K + k0);
        acc[r] = fmaf(w[0], x.x, acc[r]);
        acc[r] = fmaf(w[1], x.y, acc[r]);
        acc[r] = fmaf(w[2], x.z, acc[r]);
        acc[r] = fmaf(w[3], x.w, acc[r]);
      }
    }
  }
#pragma unroll
  for (int r = 0; r < kMTile; ++r) acc[r] = warp_sum(acc[r]);
}

// Stage rows m0..m0+mt of the (optionally LayerNorm-ed) input into shared memory, rounded
// to the weight type.  CTA 0 also writes the fp32 normalised rows to x_store.
template <typename W>
__device__ void stage_x(const GemmArgs<W>& g, float eps, int m0, int mt, W* xs) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int K = g.K;
  for (int r = warp; r < mt; r += kWarps) {
    const float* src = g.x_src + (size_t)(m0 + r) * K;
    float mean = 0.f, rstd = 1.f;
    if (g.x_g != nullptr) {
      float s = 0.f;
      for (int e = lane; e < K; e += 32) s += __ldcg(src + e);
      mean = warp_sum(s) / K;
      float s2 = 0.f;
      for (int e = lane; e < K; e += 32) { const float c = __ldcg(src + e) - mean; s2 += c * c; }
      rstd = 1.0f / sqrtf(warp_sum(s2) / K + eps);
    }
    const bool store = g.x_store != nullptr && blockIdx.x == 0;
    for (int e = lane; e < K; e += 32) {
      float v = __ldcg(src + e);
      if (g.x_g != nullptr) v = (v - mean) * rstd * to_f(g.x_g[e]) + to_f(g.x_b[e]);
      if (store) g.x_store[(size_t)(m0 + r) * K + e] = v;
      xs[(size_t)r * K + e] = from_f<W>(v);
    }
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

template <typename W>
__device__ void gemm_phase(const GemmArgs<W>& g, const Dims& D, unsigned char* smem) {
  W* xs = reinterpret_cast<W*>(smem);
  Partial* ps = reinterpret_cast<Partial*>(smem + (size_t)kMTile * (D.d > D.f ? D.d : D.f) *
                                                      sizeof(W));
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int gw = blockIdx.x * kWarps + warp;
  const int tw = gridDim.x * kWarps;
  for (int m0 = 0; m0 < g.M; m0 += kMTile) {
    const int mt = g.M - m0 < kMTile ? g.M - m0 : kMTile;
    __syncthreads();
    stage_x(g, D.eps, m0, mt, xs);
    __syncthreads();
    float amx = -INFINITY, asum = 0.f;
    int aidx = 0x7fffffff, anan = 0;
    for (int n = gw; n < g.N; n += tw) {
      float acc[kMTile];
      dot_col(g.w + (size_t)n * g.K, xs, g.K, mt, acc);
      // lane r finishes row r (a compile-time-indexed select keeps acc in registers)
      float a = 0.f;
#pragma unroll
      for (int r = 0; r < kMTile; ++r)
        if (lane == r) a = acc[r];
      if (lane < mt) {
      const int m = m0 + lane;
      const float bias = g.bias != nullptr ? to_f(g.bias[n]) : 0.f;
      const float v = a + bias;
      switch (g.epi) {
        case EPI_STORE: g.out[(size_t)m * g.ld + n] = v; break;
        case EPI_ACT: g.out[(size_t)m * g.ld + n] = act_fn(v, D.act); break;
        case EPI_RESID:
          g.out[(size_t)m * g.ld + n] = v + __ldcg(g.resid + (size_t)m * g.ld + n);
          break;
        case EPI_QKV: {
          const int which = n / D.d, c = n - which * D.d;
          if (which == 0) {
            g.out[(size_t)m * D.d + c] = v;
          } else if (g.kdst != nullptr) {
            W* dst = which == 1 ? g.kdst : g.vdst;
            dst[(size_t)(g.slot0 + m) * D.d + c] = from_f<W>(v);
          } else {
            float* dst = which == 1 ? g.kdst_f : g.vdst_f;
            dst[(size_t)m * D.d + c] = v;
          }
          break;
        }
        case EPI_KVCROSS: {
          const int layer = n / (2 * D.d), c2 = n - layer * 2 * D.d;
          const int which = c2 / D.d, c = c2 - which * D.d;
          W* dst = (which == 0 ? g.kdst : g.vdst) + (size_t)layer * g.kv_ld * D.d;
          dst[(size_t)m * D.d + c] = from_f<W>(v);
          break;
        }
        case EPI_ARGMAX: argmax_push(v, n, amx, aidx, asum, anan); break;
        case EPI_LOGITS: g.out[(size_t)m * g.ld + n] = v; break;
      }
      }
    }
    if (g.epi == EPI_ARGMAX) {
      // combine the warps of this CTA in warp order, then publish the CTA partial per row
      if (lane < kMTile) ps[warp * kMTile + lane] = Partial{amx, aidx, asum, anan};
      __syncthreads();
      if (warp == 0 && lane < mt) {
        Partial acc = ps[lane];
        for (int w2 = 1; w2 < kWarps; ++w2) partial_merge(acc, ps[w2 * kMTile + lane]);
        g.part[(size_t)blockIdx.x * g.part_ld + m0 + lane] = acc;
      }
    }
  }
}

// ------------------------------------------------------------------------------------------
// attention: out[m, head] = softmax(q k^T / sqrt(dh)) v over keys 0..T(m)-1
// ------------------------------------------------------------------------------------------

template <typename KV>
__device__ __forceinline__ float key_dot(const KV* krow, const float* qs, int dh);

template <>
__device__ __forceinline__ float key_dot<__nv_bfloat16>(const __nv_bfloat16* krow,
                                                        const float* qs, int dh) {
  float s = 0.f;
  for (int e = 0; e < dh; e += 8) {
    float k[8];
    unpack8(__ldcg(reinterpret_cast<const uint4*>(krow + e)), k);
#pragma unroll
    for (int t = 0; t < 8; ++t) s = fmaf(qs[e + t], k[t], s);
  }
  return s;
}

template <>
__device__ __forceinline__ float key_dot<float>(const float* krow, const float* qs, int dh) {
  float s = 0.f;
  for (int e = 0; e < dh; e += 4) {
    const float4 k = __ldcg(reinterpret_cast<const float4*>(krow + e));
    s = fmaf(qs[e], k.x, s);
    s = fmaf(qs[e + 1], k.y, s);
    s = fmaf(qs[e + 2], k.z, s);
    s = fmaf(qs[e + 3], k.w, s);
  }
  return s;
}

__device__ __forceinline__ float ld_kv(const float* p) { return __ldcg(p); }
__device__ __forceinline__ float ld_kv(const __nv_bfloat16* p) {
  const unsigned short u = __ldcg(reinterpret_cast<const unsigned short*>(p));
  return __uint_as_float(((unsigned)u) << 16);
}

// causal_pos0 >= 0: row m attends keys 0..causal_pos0+m; else all n_keys keys.
template <typename KV>
__device__ void attn_phase(const Dims& D, const float* q, const KV* kc, const KV* vc,
                           float* out, int M, int causal_pos0, int n_keys, float* scratch) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int gw = blockIdx.x * kWarps + warp;
  const int tw = gridDim.x * kWarps;
  const int dh = D.dh;
  float* qs = scratch + (size_t)warp * (128 + D.rows + 4);
  float* ps = qs + 128;
  const float scale = 1.0f / sqrtf((float)dh);
  for (int it = gw; it < M * D.H; it += tw) {
    const int m = it / D.H, h = it - m * D.H;
    const int T = causal_pos0 >= 0 ? causal_pos0 + m + 1 : n_keys;
    for (int e = lane; e < dh; e += 32) qs[e] = __ldcg(q + (size_t)m * D.d + h * dh + e) * scale;
    __syncwarp();
    float lmax = -INFINITY;
    for (int j = lane; j < T; j += 32) {
      const float s = key_dot<KV>(kc + (size_t)j * D.d + h * dh, qs, dh);
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
    __syncwarp();
    for (int e = lane; e < dh; e += 32) {
      float acc = 0.f;
      const KV* vp = vc + h * dh + e;
      for (int j = 0; j < T; ++j) acc = fmaf(ps[j], ld_kv(vp + (size_t)j * D.d), acc);
      out[(size_t)m * D.d + h * dh + e] = acc / sum;
    }
    __syncwarp();
  }
}

}  // namespace pd

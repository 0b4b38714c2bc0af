// cl_pass.cuh — the cluster engine (PD_ENGINE_CLUSTER): one decoder pass as three
// super-phases per layer, each run by thread-block clusters of D.cl CTAs that exchange rows
// through distributed shared memory, with a single grid barrier per super-phase.
//
// The SIMT engine separates the 8 steps of a decoder layer (QKV, self-attention, O, cross-Q,
// cross-attention, cross-O, FFN1, FFN2) by grid barriers because each step needs whole rows of
// the previous one.  Most of those dependencies are local to one attention head or to one
// slice of the FFN's hidden units, which is what the super-phases use:
//
//   SA(l)  per head h:  stage + LayerNorm, q/k/v of head h (Eq. 3's f at layer l), block-causal
//          attention of head h over the paged cache, and head h's share of the output
//          projection, attn_h . Wo[:, h]^T, written as partial sum h;
//   SB(l)  per head h:  the same for cross-attention over the cached encoder keys / values;
//   SC(l)  per hidden slice c:  FFN1 of the slice's units, activation, and the slice's share
//          of FFN2, written as partial sum c;
//
// and the next super-phase's staging adds the residual rows, the partial sums (in ascending
// order) and the bias.  Head h is worked on by cluster h mod (clusters), slice c by cluster c;
// inside a cluster the products of a step are divided over its CTAs, and the step's output
// rows are stored into every CTA's shared memory (st.shared::cluster) before a cluster barrier.
// The LM head runs over the whole grid as in the SIMT engine, each cluster staging the final
// rows for its CTAs.  Per layer that is 3 grid barriers instead of 8.
//
// Arithmetic is fp32 on the CUDA cores with the same rounding points as the SIMT engine
// (sublayer inputs, attention outputs and FFN hidden rows rounded to the weight type), but in
// a different order, so the engine is a property of the context.  Every value's summation
// order depends only on the model's shapes and the key count of its row, never on the number
// of rows in the pass or on a row's place among them: passes stay batch-invariant and every
// method returns the GPU's greedy tokens bit for bit.
#pragma once

#include "pd_device.cuh"

namespace pd {

constexpr int kClMax = 8;           // CTAs per cluster: 2, 4 or 8 (Dims::cl; 8 = portable max)
constexpr int kClRows = kMTile;     // rows per tile (the 4 x 8 reduce-scatter layout)

// ---- cluster primitives ------------------------------------------------------------------

__device__ __forceinline__ unsigned cl_rank() {
  unsigned r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ unsigned cl_index() {
  unsigned r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ unsigned cl_count() {
  unsigned r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
// Every thread of every CTA of the cluster: release / acquire at cluster scope.
__device__ __forceinline__ void cl_sync() {
  asm volatile(
      "barrier.cluster.arrive.release.aligned;\n\t"
      "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// The address of shared variable p in the shared memory of CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t cl_map(const void* p, unsigned rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
               : "=r"(r)
               : "r"((uint32_t)__cvta_generic_to_shared(p)), "r"(rank));
  return r;
}
__device__ __forceinline__ void cl_st(uint32_t a, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(a), "f"(v) : "memory");
}
__device__ __forceinline__ void cl_st(uint32_t a, __nv_bfloat16 v) {
  asm volatile("st.shared::cluster.u16 [%0], %1;" ::"r"(a), "h"(__bfloat16_as_ushort(v))
               : "memory");
}
__device__ __forceinline__ void cl_st4(uint32_t a, float4 v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(a), "f"(v.x), "f"(v.y),
               "f"(v.z), "f"(v.w)
               : "memory");
}
__device__ __forceinline__ int cl_ld_s32(uint32_t a) {
  int v;
  asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
  return v;
}
// Store v (rounded to T) at shared address p of every CTA of the cluster (ncl CTAs).
template <typename T>
__device__ __forceinline__ void cl_bcast(T* p, float v, int ncl) {
  const T t = from_f<T>(v);
  for (int r = 0; r < ncl; ++r) cl_st(cl_map(p, (unsigned)r), t);
}

// All CTAs of the grid meet.  The cluster meets first (its CTAs' writes released at cluster
// scope), then CTA 0 of every cluster fences at GPU scope, arrives on the grid counter and
// polls it (bounded, as grid_barrier), and the cluster meets again; every CTA then reads CTA
// 0's verdict, so all CTAs of a cluster take the same branch (a CTA that left early would
// leave its partners waiting at their next cluster barrier).  `during()` runs on every thread
// between the two cluster barriers.
template <typename F>
__device__ __forceinline__ bool cl_grid_barrier(unsigned* bar, unsigned& target, int* status,
                                                F&& during) {
  __shared__ int s_ok;
  cl_sync();
  target += cl_count();
  const bool lead = cl_rank() == 0 && threadIdx.x == 0;
  if (lead) {
    __threadfence();
    red_release_add(bar, 1u);
  }
  during();
  if (lead) {
    s_ok = spin_until(bar, bar, target, status);
    __threadfence();
  }
  cl_sync();
  return cl_ld_s32(cl_map(&s_ok, 0)) != 0;
}
__device__ __forceinline__ bool cl_grid_barrier(unsigned* bar, unsigned& target, int* status) {
  return cl_grid_barrier(bar, target, status, [] {});
}

// ---- products ------------------------------------------------------------------------------

// Weight row of output j of a product: w + (base + (j / seg) * sstride + j % seg) * ldw + coff
// (seg / sstride describe the interleaved q / k / v rows of one head in the fused projection;
// coff a column window, such as one head's columns of an output projection).  Groups of 4
// outputs start at multiples of 4 and seg is a multiple of 4, so a group's rows are
// consecutive rows of w.
template <typename W>
struct ClRows {
  const W* w;
  int ldw, base, seg, sstride, coff;
  __device__ __forceinline__ const W* row(int j) const {
    return w + (size_t)(base + (j / seg) * sstride + (j - (j / seg) * seg)) * ldw + coff;
  }
};

// Partial dot products of 4 consecutive weight rows (w0 + c * ldw, c < nvalid) with up to 8
// staged rows (xs + r * ldx, r < mt) over the 16-byte chunks j0..j1-1 of K: lane l sums chunks
// l, l + 32, ... in ascending order (two per lane in flight), then the reduce-scatter leaves
// (c, r) on lane c * 8 + r.
template <typename W>
__device__ __forceinline__ float cl_dot(const W* w0, int ldw, int nvalid, int j0, int j1,
                                        const W* xs, int ldx, int mt) {
  constexpr int E = 16 / (int)sizeof(W);
  const int lane = threadIdx.x & 31;
  float acc[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) acc[i] = 0.f;
  for (int j = j0 + lane; j < j1; j += 32) {
    uint4 wr[kNCol];
#pragma unroll
    for (int c = 0; c < kNCol; ++c)
      wr[c] = c < nvalid ? ldg_nc_v4(w0 + (size_t)c * ldw + (size_t)j * E)
                         : make_uint4(0u, 0u, 0u, 0u);
    if constexpr (sizeof(W) == 2) {
      float wv[kNCol][8];
#pragma unroll
      for (int c = 0; c < kNCol; ++c) unpack8(wr[c], wv[c]);
#pragma unroll
      for (int r = 0; r < kMTile; ++r) {
        if (r < mt) {
          float x[8];
          unpack8(*reinterpret_cast<const uint4*>(xs + (size_t)r * ldx + (size_t)j * E), x);
#pragma unroll
          for (int c = 0; c < kNCol; ++c)
#pragma unroll
            for (int e = 0; e < 8; ++e)
              acc[c * kMTile + r] = fmaf(wv[c][e], x[e], acc[c * kMTile + r]);
        }
      }
    } else {
#pragma unroll
      for (int r = 0; r < kMTile; ++r) {
        if (r < mt) {
          const float4 x = *reinterpret_cast<const float4*>(xs + (size_t)r * ldx + (size_t)j * E);
#pragma unroll
          for (int c = 0; c < kNCol; ++c) {
            float& a = acc[c * kMTile + r];
            a = fmaf(__uint_as_float(wr[c].x), x.x, a);
            a = fmaf(__uint_as_float(wr[c].y), x.y, a);
            a = fmaf(__uint_as_float(wr[c].z), x.z, a);
            a = fmaf(__uint_as_float(wr[c].w), x.w, a);
          }
        }
      }
    }
  }
  return reduce_scatter32(acc);
}

// Short dot products (K of at most 32 chunks): lane c * 8 + r computes output (c, r) alone,
// summing its K elements in ascending order (the weight row's loads all in flight).
template <typename W>
__device__ __forceinline__ float cl_dot_short(const W* w0, int ldw, int nvalid, int nch,
                                              const W* xs, int ldx, int mt) {
  const int lane = threadIdx.x & 31;
  const int c = lane / kMTile, r = lane % kMTile;
  float a = 0.f;
  if (c >= nvalid || r >= mt) return a;
  const uint4* wp = reinterpret_cast<const uint4*>(w0 + (size_t)c * ldw);
  const uint4* xp = reinterpret_cast<const uint4*>(xs + (size_t)r * ldx);
  for (int j0 = 0; j0 < nch; j0 += 8) {
    uint4 wr[8];
#pragma unroll
    for (int t = 0; t < 8; ++t)
      if (j0 + t < nch) wr[t] = ldg_nc_v4(wp + j0 + t);
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      if (j0 + t < nch) {
        const uint4 xv = xp[j0 + t];
        if constexpr (sizeof(W) == 2) {
          float w[8], x[8];
          unpack8(wr[t], w);
          unpack8(xv, x);
#pragma unroll
          for (int e = 0; e < 8; ++e) a = fmaf(w[e], x[e], a);
        } else {
          a = fmaf(__uint_as_float(wr[t].x), __uint_as_float(xv.x), a);
          a = fmaf(__uint_as_float(wr[t].y), __uint_as_float(xv.y), a);
          a = fmaf(__uint_as_float(wr[t].z), __uint_as_float(xv.z), a);
          a = fmaf(__uint_as_float(wr[t].w), __uint_as_float(xv.w), a);
        }
      }
    }
  }
  return a;
}

// Warps per output group of a product with ngroups groups of 4 outputs over nct CTAs and K
// (chunks of 16 bytes): enough to keep the CTA's warps busy, at most one chunk per lane.  A
// function of the shapes only.
__device__ __forceinline__ int cl_kw(int ngroups, int nch, int nct) {
  const int per_cta = (ngroups + nct - 1) / nct;
  int kw = kWarps / (per_cta > 0 ? per_cta : 1);
  const int cap = nch / 32 > 1 ? nch / 32 : 1;
  kw = kw < cap ? kw : cap;
  return kw < 1 ? 1 : (kw > kWarps ? kWarps : kw);
}

// What a cluster-engine product does with its outputs (ClGemm::epi).
enum ClEpi : int {
  CL_QKV = 0,      // v + bias: q (scaled) into every CTA's qs; k / v into the paged cache
  CL_Q = 1,        // v + bias, scaled, into every CTA's qs
  CL_PART = 2,     // partial sum: gout[(m0 + r) * d + n]
  CL_HID = 3,      // act(v + bias), rounded to W, into every CTA's hs
  CL_LOGITS = 4,   // raw logits[(m0 + r) * V + n]
  CL_ARGMAX = 5    // LM head: running argmax / max / sum of exp, merged into part[cta][row]
};

// One product of the cluster engine and its epilogue.
template <typename W>
struct ClGemm {
  int N, K, mt, m0;
  ClRows<W> wr;
  const W* xs;
  int ldx;
  int nct, cta, ncl;        // CTAs sharing the outputs, this one, CTAs of the cluster
  int epi;
  const W* bias;            // output n's bias at bias[n] (CL_QKV: the fused q / k / v bias)
  int d, dh, hoff;          // CL_QKV / CL_Q: model width, head width, head column offset
  float scale;
  float* qs;                // [8][dh] (shared)
  W *kdst, *vdst;           // CL_QKV: cache rows slot[m] (this layer)
  const int* slot;
  float* gout;              // CL_PART: this partial sum's rows
  W* hs;                    // CL_HID: [8][ldh] (shared)
  int ldh, act;
  float* logits;            // CL_LOGITS: [rows][V]
  Partial* part;            // CL_ARGMAX: [grid][part_ld]
  int part_ld;
};

// Outputs (n, r), n < N, r < mt, of sum_k wr.row(n)[k] * xs[r][k], k < K, by nct CTAs (this one
// is cta), with epilogue EPI (a compile-time choice, so each call site carries only its own):
// group g of outputs 4g..4g+3 goes to CTA g mod nct and, within it, to warp slot (g / nct) mod
// gpc; its K chunks are split into kw contiguous ranges, one per warp, whose sums are added in
// warp order.  Every thread of the CTA calls this.  red: [kWarps][32] floats and as many ints
// (or [kWarps][32] Partials for CL_ARGMAX) of shared memory.
template <typename W, int EPI, bool SHORT>
__device__ __forceinline__ void cl_gemm(const ClGemm<W>& g, float* red) {
  constexpr int E = 16 / (int)sizeof(W);
  constexpr bool argmax = EPI == CL_ARGMAX;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int ngroups, nch, kw, nct, cta, N, mt;
  {
    N = g.N; mt = g.mt; nct = g.nct; cta = g.cta;
    ngroups = (N + kNCol - 1) / kNCol;
    nch = g.K / E;
    kw = SHORT ? 1 : cl_kw(ngroups, nch, nct);
  }
  const int gpc = kWarps / kw;
  const int slot = warp / kw, part = warp - slot * kw;
  const int j0 = part * nch / kw, j1 = (part + 1) * nch / kw;
  float amx = -INFINITY, asum = 0.f;
  int aidx = 0x7fffffff, anan = 0;
  for (int base = 0; base < ngroups; base += nct * gpc) {
    const int gi = base + slot * nct + cta;
    const bool active = slot < gpc && gi < ngroups;
    const int n0 = gi * kNCol;
    const int nvalid = active ? (N - n0 < kNCol ? N - n0 : kNCol) : 0;
    float a = 0.f;
    if (active)
      a = SHORT ? cl_dot_short<W>(g.wr.row(n0), g.wr.ldw, nvalid, nch, g.xs, g.ldx, mt)
                : cl_dot<W>(g.wr.row(n0), g.wr.ldw, nvalid, j0, j1, g.xs, g.ldx, mt);
    if (kw > 1) {
      if (active) red[warp * 32 + lane] = a;
      __syncthreads();
      if (active && part == 0)
        for (int q = 1; q < kw; ++q) a += red[(warp + q) * 32 + lane];
      __syncthreads();
    }
    const int c = lane / kMTile, r = lane % kMTile;
    const bool valid = active && part == 0 && r < mt && c < nvalid;
    if constexpr (argmax) {
      if (valid) argmax_push(a, n0 + c, amx, aidx, asum, anan);
    } else {
      // the epilogue runs after a barrier, one thread per value of this round, reading its
      // arguments from shared memory there (nothing of it stays live across the products)
      int* okf = reinterpret_cast<int*>(red + kWarps * 32);
      red[warp * 32 + lane] = a;
      okf[warp * 32 + lane] = valid;
      __syncthreads();
      {
        const int w2 = threadIdx.x >> 5, l2 = threadIdx.x & 31;
        const float v0 = red[threadIdx.x];
        const int s2 = w2 / kw;
        const int n = (base + s2 * nct + cta) * kNCol + l2 / kMTile, m = g.m0 + l2 % kMTile;
        if (okf[threadIdx.x]) {
          float v = v0;
          if constexpr (EPI == CL_QKV) {
            const int w = n / g.dh, e = n - w * g.dh;
            v += to_f(g.bias[w * g.d + g.hoff + e]);
            if (w == 0) {
              cl_bcast(g.qs + (l2 % kMTile) * g.dh + e, v * g.scale, g.ncl);
            } else {
              W* dst = (w == 1 ? g.kdst : g.vdst) + (size_t)g.slot[m] * g.d + g.hoff + e;
              *dst = from_f<W>(v);
            }
          } else if constexpr (EPI == CL_Q) {
            cl_bcast(g.qs + (l2 % kMTile) * g.dh + n, (v + to_f(g.bias[n])) * g.scale, g.ncl);
          } else if constexpr (EPI == CL_PART) {
            g.gout[(size_t)m * g.d + n] = v;
          } else if constexpr (EPI == CL_HID) {
            cl_bcast(g.hs + (l2 % kMTile) * g.ldh + n, act_fn(v + to_f(g.bias[n]), g.act), g.ncl);
          } else if constexpr (EPI == CL_LOGITS) {
            g.logits[(size_t)m * g.N + n] = v;
          }
        }
      }
      __syncthreads();
    }
  }
  if constexpr (argmax) {
    // lane c*8 + r holds row r over its columns 4g + c; a row's partials are merged in
    // (warp, column) order, then by a fixed butterfly (as gemm_phase)
    Partial* ps = reinterpret_cast<Partial*>(red);
    __syncthreads();
    ps[warp * 32 + lane] = Partial{amx, aidx, asum, anan};
    __syncthreads();
    for (int rr = warp; rr < mt; rr += kWarps) {
      Partial acc{-INFINITY, 0x7fffffff, 0.f, 0};
      for (int e = lane; e < kWarps * kNCol; e += 32)
        partial_merge(acc, ps[(e / kNCol) * 32 + (e % kNCol) * kMTile + rr]);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) partial_merge(acc, shfl_partial(acc, o));
      if (lane == 0) g.part[(size_t)g.cta * g.part_ld + g.m0 + rr] = acc;
    }
    __syncthreads();
  }
}

// ---- staging -------------------------------------------------------------------------------

// The rows a super-phase starts from: y = r_in + (sum_p part[p] + bias), the partial sums in
// ascending p; or, for layer 0, the embedding of the rows' tokens.  ln_a (if any) turns y into
// the new residual stream, stored to r_out by cluster 0; ln_b (if any) turns that into the
// sublayer input.
template <typename W>
struct ClStage {
  const float* r_in;
  const float* part;
  int np;
  size_t part_ld;           // floats between partial sums (rows * d)
  const W* bias;
  int emb;
  const W *lna_g, *lna_b;
  float* r_out;
  const W *lnb_g, *lnb_b;
};

// Sum of partial sums p0..p1-1 of one float4 item (ascending p, 4 loads in flight).
__device__ __forceinline__ float4 cl_sum_parts(const float* part, size_t part_ld, size_t o,
                                               int p0, int p1) {
  float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int pb = p0; pb < p1; pb += 4) {
    float4 v[4];
#pragma unroll
    for (int t = 0; t < 4; ++t)
      if (pb + t < p1)
        v[t] = __ldcg(reinterpret_cast<const float4*>(part + (size_t)(pb + t) * part_ld + o));
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      if (pb + t < p1) {
        s.x += v[t].x; s.y += v[t].y; s.z += v[t].z; s.w += v[t].w;
      }
    }
  }
  return s;
}

// y = rr + (s + bias) of one float4 item, stored into every CTA's ys.
template <typename W>
__device__ __forceinline__ void cl_stage_put(const ClStage<W>& a, const Dims& D, float4 s,
                                             float4 rr, int k, float* dst) {
  if (a.bias != nullptr) {
    const float4 b = get4(a.bias + k);
    s.x += b.x; s.y += b.y; s.z += b.z; s.w += b.w;
  }
  const float4 y = make_float4(rr.x + s.x, rr.y + s.y, rr.z + s.z, rr.w + s.w);
  for (int c = 0; c < D.cl; ++c) cl_st4(cl_map(dst, (unsigned)c), y);
}

// This CTA's d / D.cl features of tile rows m0..m0+mt-1: y = r_in + (sum_p part[p] + bias),
// stored into every CTA's ys (fp32).  When a full tile has fewer 4-feature items than the CTA
// has threads, the partial sums of an item are split into nq contiguous ranges summed by nq
// threads (ascending p within a range, the ranges added in order); nq depends on d and the
// cluster size only, so a row's sum does not depend on the rows the tile carries.
// red: blockDim.x float4 of shared memory.
template <typename W>
__device__ __forceinline__ void cl_stage_sum(const ClStage<W>& a, const Dims& D, int m0, int mt,
                                             float* ys, float* red) {
  const int d = D.d;
  const int w4 = d / (4 * D.cl), k0 = (int)cl_rank() * (d / D.cl);
  const int items_max = kClRows * w4;             // float4 items of a full tile
  const int nq = (int)blockDim.x / items_max;
  if (nq <= 1) {
    for (int it = threadIdx.x; it < mt * w4; it += blockDim.x) {
      const int r = it / w4, k = k0 + (it - r * w4) * 4;
      const size_t o = (size_t)(m0 + r) * d + k;
      const float4 rr = __ldcg(reinterpret_cast<const float4*>(a.r_in + o));
      cl_stage_put(a, D, cl_sum_parts(a.part, a.part_ld, o, 0, a.np), rr, k, ys + (size_t)r * d + k);
    }
    return;
  }
  const int it = threadIdx.x % items_max, q = threadIdx.x / items_max;
  const int r = it / w4, k = k0 + (it - r * w4) * 4;
  const size_t o = (size_t)(m0 + r) * d + k;
  float4* red4 = reinterpret_cast<float4*>(red);
  float4 rr = make_float4(0.f, 0.f, 0.f, 0.f);
  if (q == 0 && r < mt) rr = __ldcg(reinterpret_cast<const float4*>(a.r_in + o));
  if (q < nq && r < mt)
    red4[q * items_max + it] = cl_sum_parts(a.part, a.part_ld, o, q * a.np / nq, (q + 1) * a.np / nq);
  __syncthreads();
  if (q == 0 && r < mt) {
    float4 s = red4[it];
    for (int qq = 1; qq < nq; ++qq) {
      const float4 t = red4[qq * items_max + it];
      s.x += t.x; s.y += t.y; s.z += t.z; s.w += t.w;
    }
    cl_stage_put(a, D, s, rr, k, ys + (size_t)r * d + k);
  }
}

// LayerNorm of the row y[0..d) (shared memory, fp32) by one warp, in place (ln_regs: mean and
// biased variance from per-lane sums over elements lane * 4 + 128 i, fixed butterflies).
template <typename W>
__device__ __forceinline__ void cl_ln_row(float* y, int d, const W* g, const W* b, float eps) {
  const int lane = threadIdx.x & 31;
  const int nI = d / 128;
  float4 v[kMaxRowRegs];
#pragma unroll
  for (int i = 0; i < kMaxRowRegs; ++i)
    if (i < nI) v[i] = *reinterpret_cast<const float4*>(y + lane * 4 + 128 * i);
  ln_regs(v, nI, d, g, b, eps);
#pragma unroll
  for (int i = 0; i < kMaxRowRegs; ++i)
    if (i < nI) *reinterpret_cast<float4*>(y + lane * 4 + 128 * i) = v[i];
  __syncwarp();
}

// Embedding of token t at position p (E[t] * sqrt(d) + position row) into y (shared memory,
// fp32) by one warp, every load of the row in flight before the stores.  Not inlined: it runs
// once per pass, and its registers stay out of the products' loops.
template <typename W>
__device__ __noinline__ void cl_embed_row(const EmbedTabs<W>& T, const Dims& D, int t, int p,
                                          float* y) {
  const int lane = threadIdx.x & 31;
  const int d = D.d;
  t = t < 0 ? 0 : (t >= D.V ? D.V - 1 : t);
  const W* er = T.E + (size_t)t * d;
  const float* pr = T.P == nullptr ? T.ptab + (size_t)p * d : nullptr;
  const W* lr = T.P != nullptr ? T.P + (size_t)(p < D.max_pos ? p : D.max_pos - 1) * d : nullptr;
  float4 e[kMaxRowRegs], ps[kMaxRowRegs];
#pragma unroll
  for (int i = 0; i < kMaxRowRegs; ++i) {
    const int k = lane * 4 + 128 * i;
    if (k < d) {
      e[i] = get4(er + k);
      ps[i] = lr != nullptr ? get4(lr + k) : *reinterpret_cast<const float4*>(pr + k);
    }
  }
#pragma unroll
  for (int i = 0; i < kMaxRowRegs; ++i) {
    const int k = lane * 4 + 128 * i;
    if (k < d)
      *reinterpret_cast<float4*>(y + k) =
          make_float4(e[i].x * D.emb_scale + ps[i].x, e[i].y * D.emb_scale + ps[i].y,
                      e[i].z * D.emb_scale + ps[i].z, e[i].w * D.emb_scale + ps[i].w);
  }
  __syncwarp();
}

// Tile rows m0..m0+mt-1 in ys (or, layer 0, their embeddings written there), one warp per row,
// in place: ln_a, the new residual row (cluster 0), ln_b, rounded into us.
template <typename W>
__device__ __forceinline__ void cl_stage_rows(const ClStage<W>& a, const EmbedTabs<W>& T,
                                              const Dims& D, const int* rtok, const int* rpos,
                                              int m0, int mt, float* ys, W* us) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int d = D.d;
  const bool writer = a.r_out != nullptr && cl_index() == 0;
  const int rank = (int)cl_rank();
  for (int r = warp; r < mt; r += kWarps) {
    const int m = m0 + r;
    float* y = ys + (size_t)r * d;
    if (a.emb) cl_embed_row(T, D, rtok[m], rpos[m], y);
    if (a.lna_g != nullptr) cl_ln_row(y, d, a.lna_g, a.lna_b, D.eps);
    if (writer && (r % D.cl) == rank)
      for (int k = lane * 4; k < d; k += 128)
        *reinterpret_cast<float4*>(a.r_out + (size_t)m * d + k) =
            *reinterpret_cast<const float4*>(y + k);
    if (a.lnb_g != nullptr) cl_ln_row(y, d, a.lnb_g, a.lnb_b, D.eps);
    for (int k = lane * 4; k < d; k += 128)
      put4(us + (size_t)r * d + k, *reinterpret_cast<const float4*>(y + k));
  }
}

// Stage tile rows m0..m0+mt-1 into every CTA of the cluster: each CTA sums its d / D.cl
// features of every row into every CTA's ys, a cluster barrier, then each CTA normalises the
// rows (one warp per row) into us (weight type).
template <typename W>
__device__ __forceinline__ void cl_stage(const ClStage<W>& a, const EmbedTabs<W>& T,
                                         const Dims& D, const int* rtok, const int* rpos, int m0,
                                         int mt, float* ys, W* us, float* red) {
  if (!a.emb) {
    cl_stage_sum(a, D, m0, mt, ys, red);
    cl_sync();
  } else {
    __syncthreads();
  }
  cl_stage_rows(a, T, D, rtok, rpos, m0, mt, ys, us);
  __syncthreads();
}

// ---- attention of one row ----------------------------------------------------------------

// One row of one head by all warps of this CTA: q (fp32, scaled by 1/sqrt(dh), in shared
// memory) against keys 0..T-1 of kc / vc at head offset hoff; key j sits at row base + j
// (contiguous cache) or, given a page table ptab ([sentence][pt_ld]), in pool page
// ptab[base][j / 16] at row j % 16.  Scores one key per thread, softmax with the CTA-wide
// maximum and a sum in thread order, value sums per warp over keys j = warp, warp + kWarps, ...
// (ascending), added in warp order.  The result (divided by the sum) is stored into row orow
// of every CTA's attention tile.
template <typename W>
__device__ __noinline__ void cl_attn_row(const Dims& D, const float* q, const W* kc, const W* vc,
                                         int hoff, int T, const int* ptab, int base, float* sc,
                                         float* wred, W* orow) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int dh = D.dh;
  constexpr int E = 16 / (int)sizeof(W);
  const int nchk = dh / E;
  float lmax = -INFINITY;
  for (int j = threadIdx.x; j < T; j += blockDim.x) {
    const uint4* kr =
        reinterpret_cast<const uint4*>(kc + key_row<W>(ptab, D.pt_ld, base, j) * D.d + hoff);
    float s = 0.f;
    for (int c0 = 0; c0 < nchk; c0 += 8) {     // 8 loads of the key row in flight
      uint4 kk[8];
#pragma unroll
      for (int c = 0; c < 8; ++c)
        if (c0 + c < nchk) kk[c] = __ldcg(kr + c0 + c);
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        if (c0 + c < nchk) {
          const float* qc = q + (c0 + c) * E;
          if constexpr (sizeof(W) == 2) {
            float k[8];
            unpack8(kk[c], k);
#pragma unroll
            for (int t = 0; t < 8; ++t) s = fmaf(qc[t], k[t], s);
          } else {
            s = fmaf(qc[0], __uint_as_float(kk[c].x), s);
            s = fmaf(qc[1], __uint_as_float(kk[c].y), s);
            s = fmaf(qc[2], __uint_as_float(kk[c].z), s);
            s = fmaf(qc[3], __uint_as_float(kk[c].w), s);
          }
        }
      }
    }
    sc[j] = s;
    lmax = fmaxf(lmax, s);
  }
  lmax = warp_max(lmax);
  if (lane == 0) wred[warp] = lmax;
  __syncthreads();
  float mx = wred[0];
  for (int w = 1; w < kWarps; ++w) mx = fmaxf(mx, wred[w]);
  float lsum = 0.f;
  for (int j = threadIdx.x; j < T; j += blockDim.x) {
    const float p = expf(sc[j] - mx);
    sc[j] = p;
    lsum += p;
  }
  lsum = warp_sum(lsum);
  __syncthreads();                       // every warp has read the maxima
  if (lane == 0) wred[warp] = lsum;
  __syncthreads();
  float sum = 0.f;
  for (int w = 0; w < kWarps; ++w) sum += wred[w];
  // value sums: lane covers elements lane * epl .. (epl = dh / 32 consecutive elements)
  const int epl = dh / 32;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int j0 = warp; j0 < T; j0 += 4 * kWarps) {   // 4 keys' value loads in flight
    float vv[4][4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int j = j0 + t * kWarps;
      if (j < T) {
        const W* vr = vc + key_row<W>(ptab, D.pt_ld, base, j) * D.d + hoff + lane * epl;
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (e < epl) vv[t][e] = to_f(__ldcg(vr + e));
      }
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int j = j0 + t * kWarps;
      if (j < T) {
        const float p = sc[j];
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (e < epl) acc[e] = fmaf(p, vv[t][e], acc[e]);
      }
    }
  }
  float* part = wred + 2 * kWarps;       // [kWarps][dh]
#pragma unroll
  for (int e = 0; e < 4; ++e)
    if (e < epl) part[warp * dh + lane * epl + e] = acc[e];
  __syncthreads();
  for (int e = threadIdx.x; e < dh; e += blockDim.x) {
    float t = 0.f;
    for (int w = 0; w < kWarps; ++w) t += part[w * dh + e];
    cl_bcast(orow + e, t / sum, D.cl);
  }
  __syncthreads();                       // sc and wred are free again
}

}  // namespace pd

// pd.cu — kernels and C ABI of the GB300 parallel decoder (see include/pd.h).
//
// Execution model.  One persistent, cooperatively launched kernel per pd_encode and per
// pd_decode call: one 512-thread CTA per SM.  pd_decode's kernel runs the whole decoding
// loop on the device — every decoder pass (embedding, Ld x {QKV, self-attention, O-proj,
// cross-Q, cross-attention, cross-O, FFN1, FFN2}, LM head with fused argmax) and the
// fixed-point commit that advances the block — with grid barriers between phases and no
// host round trip per pass.  The pass loop is bounded by Proposition 1 (at most m passes)
// and by the optional pass budget; every device wait is bounded in time.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstddef>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <algorithm>
#include <vector>

#include <cudaTypedefs.h>

#include "pd.h"
#include "pd_device.cuh"
#include "tc_gemm.cuh"
#include "cl_pass.cuh"

namespace pd {

template <typename W>
struct KParams {
  Dims D;
  const ModelW<W>* mw;      // device copy of the weight-pointer table
  Bufs<W> B;
  int n_src;                // encode: source length
  int enc_slot;             // encode: cache slot of the sentence (0 for pd_encode)
  const int* enc_tok;       // encoder input ids (device)
  int debug_len;            // > 0: one teacher-forced pass over dbg_tok (slot 0), logits out
  float* logits;            // [debug_len][V]
  DecState init;            // method, b, h, stop_at_eos, max_passes, stop_rule (all sentences)
  int n_sent;               // decode: sentences, slots 0..n_sent-1
  int n_src_s[kMaxBatch];   // decode: source length of each sentence
  int max_len_s[kMaxBatch]; // decode: max_len (the known m of Jacobi / GS-Jacobi) of each
  int32_t* out_y;           // [n_sent][out_ld]
  int out_ld;
  int32_t* out_info;        // [n_sent][4] = {n_y, n_iters, status, n_trace}
  // bf16: TMA tensor map of the weight matrix of every GEMM phase of this kernel's sequence
  CUtensorMap maps[kMaxKernelMaps];
};

// Dynamic shared memory of the decode / encode kernels (byte offsets): xs, the staged GEMM
// input rows (8 rows x max(d, f) in the weight type); part, the LM head's per-warp argmax
// partials; scratch, the attention phase's per-warp scaled query and scores; commit, the
// decoding state of this CTA (see CommitMem); ln, the copied LayerNorm vectors and biases
// (ln_bytes, possibly 0).
struct SmemLayout {
  size_t xs, part, scratch, commit, ln, ln_bytes, total;
  // bf16 (tensor-core) kernels: weight slots, staged token rows, epilogue tile; all offsets
  // are relative to the first 1024-byte aligned address of the dynamic shared memory, and
  // total includes the 1024 bytes of alignment slack
  size_t ring, bbuf, epi;
  int ring_slots;
  // cluster-engine kernels (cl_pass.cuh): xs holds the staged fp32 rows of a tile; us the
  // sublayer inputs, qs the tile's scaled queries, as its attention outputs, hs its FFN hidden
  // units (part holds the products' warp sums and the LM head's partials; scratch the
  // attention scores and warp sums)
  size_t us, qs, as, hs;
};

// The commit region: per pass row r (at most D.rows) its new token (-1 for a NaN row) and
// probability, and the row's description (input token, position, self-attention cache slot,
// its sentence, keys it attends, first cross key row and cross key count); per sentence its
// decoding state, its first row in the pass, y_0..y_m and its page table (the pool page of
// each 16 positions of its self-attention keys and values).
struct CommitMem {
  int *ntok, *rtok, *rpos, *rslot, *rsb, *rkn, *rxb, *rxn;
  float* nprob;
  DecState* st;
  int* r0;
  int* y;                   // [max_batch][max_tgt + 1]
  int* pt;                  // [max_batch][pt_ld]
  int* misc;                // [0] rows of the current pass
};
__host__ __device__ inline size_t commit_bytes(const Dims& D) {
  return (size_t)D.rows * 9 * 4 + (size_t)D.max_batch * (sizeof(DecState) + 4) +
         (size_t)D.max_batch * (D.max_tgt + 1) * 4 + (size_t)D.max_batch * D.pt_ld * 4 + 64;
}

// Cache slot of position pos of the sentence whose page table is pt.
__device__ __forceinline__ int page_slot(const int* pt, int pos) {
  return pt[pos >> kPageShift] * kPageRows + (pos & (kPageRows - 1));
}
__device__ __forceinline__ CommitMem commit_mem(const Dims& D, unsigned char* base) {
  CommitMem c;
  int* p = reinterpret_cast<int*>(base);
  c.ntok = p; p += D.rows;
  c.rtok = p; p += D.rows;
  c.rpos = p; p += D.rows;
  c.rslot = p; p += D.rows;
  c.rsb = p; p += D.rows;
  c.rkn = p; p += D.rows;
  c.rxb = p; p += D.rows;
  c.rxn = p; p += D.rows;
  c.nprob = reinterpret_cast<float*>(p); p += D.rows;
  c.st = reinterpret_cast<DecState*>(p); p += D.max_batch * (int)(sizeof(DecState) / 4);
  c.r0 = p; p += D.max_batch;
  c.y = p; p += D.max_batch * (D.max_tgt + 1);
  c.pt = p; p += D.max_batch * D.pt_ld;
  c.misc = p;
  return c;
}

// The decoder's small vectors kept in shared memory: the LayerNorm vectors (per layer ln1,
// ln2, ln3 gamma / beta, and the embedding and final LayerNorms of pre-LN models) when they fit
// in kVecSmemMax bytes, and with them the biases (per layer qkv, o, cross-q, cross-o, ffn1,
// ffn2) when both fit.  Per layer, in elements: 6 d of LayerNorm, then 7 d + f of bias.
constexpr size_t kVecSmemMax = 112 * 1024;
__host__ __device__ inline size_t ln_elems(const Dims& D) {
  return ((size_t)D.Ld * 6 + (D.pre_ln ? 4 : 0)) * D.d;
}
__host__ __device__ inline size_t bias_elems(const Dims& D) {
  return (size_t)D.Ld * (7 * (size_t)D.d + D.f);
}
__host__ __device__ inline size_t vec_smem_bytes(const Dims& D, size_t wsize) {
  const size_t ln = ln_elems(D) * wsize, all = ln + bias_elems(D) * wsize;
  return all <= kVecSmemMax ? all : (ln <= kVecSmemMax ? ln : 0);
}

constexpr size_t kSmemMax = 227 * 1024;    // dynamic shared memory of one CTA
constexpr size_t kSmemStatic = 8 * 1024;   // reserve for the kernels' static shared memory

__host__ __device__ inline SmemLayout smem_layout(const Dims& D, size_t wsize) {
  SmemLayout L{};
  if (wsize == 2 && D.tc) {
    // tensor-core layout: as many weight slots as fit (at most kRingMax), then the vector
    // copies if they still fit
    const size_t budget = kSmemMax - kSmemStatic - 1024;
    // attention scratch, or the LM head's running argmax partial of every row of a pass
    const size_t att = (size_t)kWarps * (128 + D.max_keys + 4) * sizeof(float);
    const size_t parts = ((size_t)D.rows * sizeof(Partial) + 15) / 16 * 16;
    const size_t scratch = att > parts ? att : parts;
    const size_t fixed = kBBytes + kEpiBytes + scratch + commit_bytes(D) + 64;
    const size_t room = budget > fixed ? (budget - fixed) / kSlotBytes : 0;
    L.ring_slots = (int)(room < (size_t)kRingMax ? room : (size_t)kRingMax);
    L.ring = 0;
    L.bbuf = (size_t)L.ring_slots * kSlotBytes;
    L.epi = L.bbuf + kBBytes;
    L.scratch = L.epi + kEpiBytes;
    L.xs = L.part = L.scratch;
    L.commit = L.scratch + scratch;
    L.ln = (L.commit + commit_bytes(D) + 15) / 16 * 16;
    const size_t all = vec_smem_bytes(D, wsize), ln = ln_elems(D) * wsize;
    L.ln_bytes = L.ln + all <= budget ? all : (L.ln + ln <= budget && ln <= kVecSmemMax ? ln : 0);
    L.total = 1024 + L.ln + L.ln_bytes;
    return L;
  }
  if (D.cl) {
    auto a16 = [](size_t b) { return (b + 15) / 16 * 16; };
    L.xs = 0;
    L.us = L.xs + a16((size_t)kClRows * D.d * 4);
    L.qs = L.us + a16((size_t)kClRows * D.d * wsize);
    L.as = L.qs + a16((size_t)kClRows * D.dh * 4);
    L.hs = L.as + a16((size_t)kClRows * D.dh * wsize);
    L.part = L.hs + a16((size_t)kClRows * D.cl_fu * D.cl * wsize);
    L.scratch = L.part + (size_t)kWarps * 32 * sizeof(Partial);
    L.commit = L.scratch + a16(((size_t)D.max_keys + 2 * kWarps + (size_t)kWarps * D.dh) * 4);
    L.ln = a16(L.commit + commit_bytes(D));
    const size_t all = vec_smem_bytes(D, wsize), ln = ln_elems(D) * wsize;
    const size_t slack = wsize == 2 ? 1024 : 0;   // smem_base's alignment of bf16 kernels
    L.ln_bytes = L.ln + all + slack <= kSmemMax ? all
                 : (L.ln + ln + slack <= kSmemMax && ln <= kVecSmemMax ? ln : 0);
    L.total = slack + L.ln + L.ln_bytes;
    return L;
  }
  const int kmax = D.d > D.f ? D.d : D.f;
  L.xs = 0;
  L.part = L.xs + ((size_t)kMTile * kmax * wsize + 15) / 16 * 16;
  L.scratch = L.part + (size_t)kWarps * 32 * sizeof(Partial);
  L.commit = L.scratch + (size_t)kWarps * (128 + D.max_keys + 4) * sizeof(float);
  L.ln = (L.commit + commit_bytes(D) + 15) / 16 * 16;
  // the vector copies are kept only when they fit beside the rest
  const size_t all = vec_smem_bytes(D, wsize), ln = ln_elems(D) * wsize;
  // bf16 kernels align their dynamic shared memory to 1024 bytes (smem_base): keep the slack
  const size_t slack = wsize == 2 ? 1024 : 0;
  L.ln_bytes = L.ln + all + slack <= kSmemMax ? all
               : (L.ln + ln + slack <= kSmemMax && ln <= kVecSmemMax ? ln : 0);
  L.total = slack + L.ln + L.ln_bytes;
  return L;
}

// ------------------------------------------------------------------------------------------
// one decoder pass over M rows (input tokens tok[0..M) at positions pos0..pos0+M-1)
// ------------------------------------------------------------------------------------------

// The weight-pointer table, copied into shared memory when a kernel starts: the acquire at
// every grid barrier drops the SM's L1 copies of global data, so a table read from global
// memory would cost an L2 round trip in every phase.
template <typename W>
__device__ __forceinline__ ModelW<W>& smem_mw() {
  __shared__ ModelW<W> s;
  return s;
}
// The model dimensions, also copied into shared memory: device functions that are not inlined
// take them by reference, and a reference into the kernel parameters or the stack would be
// read through L1, which every barrier's acquire drops.
template <typename W>
__device__ __forceinline__ Dims& smem_dims() {
  __shared__ Dims s;
  return s;
}
template <typename W>
__device__ __forceinline__ EmbedTabs<W>& smem_tabs() {
  __shared__ EmbedTabs<W> s;
  return s;
}
template <typename W>
__device__ __forceinline__ void load_smem_mw(const KParams<W>& P) {
  static_assert(sizeof(ModelW<W>) % 8 == 0, "pointer table");
  const unsigned long long* src = reinterpret_cast<const unsigned long long*>(P.mw);
  unsigned long long* dst = reinterpret_cast<unsigned long long*>(&smem_mw<W>());
  for (int i = threadIdx.x; i < (int)(sizeof(ModelW<W>) / 8); i += blockDim.x) dst[i] = src[i];
  if (threadIdx.x == 0) smem_dims<W>() = P.D;
  __syncthreads();
  if (threadIdx.x == 0) {
    const ModelW<W>& mw = smem_mw<W>();
    smem_tabs<W>() = EmbedTabs<W>{mw.embed, P.D.learned_pos ? mw.pos : nullptr,
                                  P.D.learned_pos ? nullptr : P.B.pos_tab};
  }
  __syncthreads();
}

// Copy the decoder's LayerNorm vectors (and biases, see vec_smem_bytes) into the shared-memory
// region and point the shared pointer table at the copies: a LayerNorm prologue then reads its
// gamma / beta, and an epilogue its bias, from shared memory instead of making an L2 round
// trip (every barrier's acquire drops the SM's L1 copies of global data).
template <typename W>
__device__ void load_smem_vectors(const Dims& D, unsigned char* smem) {
  const SmemLayout L = smem_layout(D, sizeof(W));
  if (L.ln_bytes == 0) return;
  const bool with_bias = L.ln_bytes > ln_elems(D) * sizeof(W);
  ModelW<W>& mw = smem_mw<W>();
  W* dst = reinterpret_cast<W*>(smem + L.ln);
  // vector v: its pointer field in the shared table and its length (elements); laid out in
  // order, LayerNorm vectors first
  const int nln = 6 * D.Ld + (D.pre_ln ? 4 : 0);
  const int nv = nln + (with_bias ? 6 * D.Ld : 0);
  auto field = [&](int v, int& len) -> const W*& {
    len = D.d;
    if (v < 6 * D.Ld) {
      DecLayerW<W>& Ly = mw.dec[v / 6];
      switch (v % 6) {
        case 0: return Ly.ln1g;
        case 1: return Ly.ln1b;
        case 2: return Ly.ln2g;
        case 3: return Ly.ln2b;
        case 4: return Ly.ln3g;
        default: return Ly.ln3b;
      }
    }
    if (v < nln) {
      switch (v - 6 * D.Ld) {
        case 0: return mw.dec_lne_g;
        case 1: return mw.dec_lne_b;
        case 2: return mw.dec_lnf_g;
        default: return mw.dec_lnf_b;
      }
    }
    DecLayerW<W>& Ly = mw.dec[(v - nln) / 6];
    switch ((v - nln) % 6) {
      case 0: len = 3 * D.d; return Ly.bqkv;
      case 1: return Ly.bo;
      case 2: return Ly.bqc;
      case 3: return Ly.boc;
      case 4: len = D.f; return Ly.b1;
      default: return Ly.b2;
    }
  };
  // every warp copies vectors v = warp, warp + kWarps, ... (16 bytes per lane and step)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  size_t off = 0;
  for (int v = 0; v < nv; ++v) {
    int len;
    const W* src = field(v, len);
    if (v % kWarps == warp && src != nullptr) {
      const int chunks = len * (int)sizeof(W) / 16;
      for (int j = lane; j < chunks; j += 32)
        *reinterpret_cast<uint4*>(reinterpret_cast<char*>(dst + off) + j * 16) =
            ldg_nc_v4(reinterpret_cast<const char*>(src) + j * 16);
    }
    off += len;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    off = 0;
    for (int v = 0; v < nv; ++v) {
      int len;
      const W*& f = field(v, len);
      if (f != nullptr) f = dst + off;
      off += len;
    }
  }
  __syncthreads();
}

// Phases of a decoder pass, per layer in this order (the attention phases take scalar
// arguments); phase 8 * Ld is the LM head.
enum : int {
  PH_QKV = 0, PH_SELF = 1, PH_O = 2, PH_QC = 3, PH_CROSS = 4, PH_OC = 5, PH_FFN1 = 6, PH_FFN2 = 7
};

__device__ __forceinline__ bool is_attn_phase(int ph, int nph) {
  return ph < nph - 1 && ((ph & 7) == PH_SELF || (ph & 7) == PH_CROSS);
}

// Arguments of GEMM phase ph of a pass over M rows, row m with input token rtok[m] at position
// rpos[m] and self-attention cache slot rslot[m]; the LM head (ph = 8 Ld) writes raw logits if
// logits != nullptr, else argmax partials.
template <typename W>
__device__ void gemm_args(const KParams<W>& P, int ph, int M, const int* rtok, const int* rpos,
                          const int* rslot, float* logits, GemmArgs<W>& g) {
  const Dims& D = smem_dims<W>();
  const Bufs<W>& B = P.B;
  const ModelW<W>& mw = smem_mw<W>();
  const bool pre = D.pre_ln != 0;
  g = GemmArgs<W>{};
  g.M = M;
  if (ph == 8 * D.Ld) {                 // LM head over the final hidden rows
    g.N = D.V; g.K = D.d; g.x_src = B.ra;
    g.ln_b_g = pre ? mw.dec_lnf_g : mw.dec[D.Ld - 1].ln3g;
    g.ln_b_b = pre ? mw.dec_lnf_b : mw.dec[D.Ld - 1].ln3b;
    g.w = mw.embed;
    if (logits != nullptr) { g.epi = EPI_LOGITS; g.out = logits; g.ld = D.V; }
    else { g.epi = EPI_ARGMAX; g.part = B.part; g.part_ld = D.rows; }
    gemm_plan(g, gridDim.x);
    return;
  }
  const int l = ph >> 3;
  const DecLayerW<W>& L = mw.dec[l];
  switch (ph & 7) {
    case PH_QKV:
      // self-attention sublayer input.  Pre-LN: x = LN1(r), residual r.  Post-LN: x = the
      // previous sublayer's LN of its output, which is also the residual; layer 0 takes the
      // embedding as is.  The embedding is computed in this GEMM's prologue.
      g.N = 3 * D.d; g.K = D.d;
      if (l == 0) {
        g.emb_tok = rtok; g.emb_pos = rpos; g.x_store = B.ra;
        if (pre) {
          g.ln_a_g = mw.dec_lne_g; g.ln_a_b = mw.dec_lne_b; g.ln_b_g = L.ln1g; g.ln_b_b = L.ln1b;
        }
      } else {
        g.x_src = B.ra;
        if (pre) { g.ln_b_g = L.ln1g; g.ln_b_b = L.ln1b; }
        else { g.ln_a_g = mw.dec[l - 1].ln3g; g.ln_a_b = mw.dec[l - 1].ln3b; g.x_store = B.xa; }
      }
      g.w = L.wqkv; g.bias = L.bqkv; g.epi = EPI_QKV; g.out = B.q; g.ld = D.d;
      g.kdst = B.kself + (size_t)l * D.kv_pages * kPageRows * D.d;
      g.vdst = B.vself + (size_t)l * D.kv_pages * kPageRows * D.d;
      g.slot = rslot;
      break;
    case PH_O:                          // self-attention output + residual
      g.N = D.d; g.K = D.d; g.xw_src = B.att; g.w = L.wo; g.bias = L.bo;
      g.epi = EPI_RESID; g.out = B.rb; g.ld = D.d; g.resid = (pre || l == 0) ? B.ra : B.xa;
      break;
    case PH_QC:                         // cross-attention query
      g.N = D.d; g.K = D.d; g.x_src = B.rb;
      if (pre) { g.ln_b_g = L.ln2g; g.ln_b_b = L.ln2b; }
      else { g.ln_a_g = L.ln1g; g.ln_a_b = L.ln1b; g.x_store = B.xb; }
      g.w = L.wqc; g.bias = L.bqc; g.epi = EPI_STORE; g.out = B.q; g.ld = D.d;
      break;
    case PH_OC:                         // cross-attention output + residual
      g.N = D.d; g.K = D.d; g.xw_src = B.att; g.w = L.woc; g.bias = L.boc;
      g.epi = EPI_RESID; g.out = B.rc; g.ld = D.d; g.resid = pre ? B.rb : B.xb;
      break;
    case PH_FFN1:
      g.N = D.f; g.K = D.d; g.x_src = B.rc;
      if (pre) { g.ln_b_g = L.ln3g; g.ln_b_b = L.ln3b; }
      else { g.ln_a_g = L.ln2g; g.ln_a_b = L.ln2b; g.x_store = B.xc; }
      g.w = L.w1; g.bias = L.b1; g.epi = EPI_ACT; g.out_w = B.ffh; g.ld = D.f;
      break;
    case PH_FFN2:
      g.N = D.d; g.K = D.f; g.xw_src = B.ffh; g.w = L.w2; g.bias = L.b2;
      g.epi = EPI_RESID; g.out = B.ra; g.ld = D.d; g.resid = pre ? B.rc : B.xc;
      break;
  }
  gemm_plan(g, gridDim.x);
}

// Ask L2 for the weight rows this CTA reads in GEMM phase ph (nothing for attention phases),
// so that HBM streams them while the latency-bound chain of earlier phases runs.
template <typename W>
__device__ void prefetch_phase(const KParams<W>& P, int ph) {
  const Dims& D = smem_dims<W>();
  const int nph = 8 * D.Ld + 1;
  if (ph >= nph || is_attn_phase(ph, nph)) return;
  const ModelW<W>& mw = smem_mw<W>();
  if (ph == nph - 1) { prefetch_gemm_weights(mw.embed, D.V, D.d); return; }
  const DecLayerW<W>& L = mw.dec[ph >> 3];
  switch (ph & 7) {
    case PH_QKV: prefetch_gemm_weights(L.wqkv, 3 * D.d, D.d); break;
    case PH_O: prefetch_gemm_weights(L.wo, D.d, D.d); break;
    case PH_QC: prefetch_gemm_weights(L.wqc, D.d, D.d); break;
    case PH_OC: prefetch_gemm_weights(L.woc, D.d, D.d); break;
    case PH_FFN1: prefetch_gemm_weights(L.w1, D.f, D.d); break;
    case PH_FFN2: prefetch_gemm_weights(L.w2, D.d, D.f); break;
  }
}

// The weights a pass reads first (phases 0 and 2) and the LM head's table, asked from L2 when
// the pass starts (the other phases' weights are asked three phases ahead).
template <typename W>
__device__ void prefetch_pass_start(const KParams<W>& P) {
  prefetch_phase(P, 0);
  prefetch_phase(P, 2);
  prefetch_phase(P, 8 * smem_dims<W>().Ld);
}

template <typename W>
__device__ __forceinline__ GemmArgs<W>& smem_args() {
  __shared__ GemmArgs<W> s;
  return s;
}

// bf16 kernels can run their GEMM phases on the tensor cores (tc_gemm.cuh), as the context
// chose (Dims::tc); fp32 kernels always run them on the SIMT path (gemm_phase).
template <typename W>
constexpr bool kTensorCores = sizeof(W) == 2;
// Kernels are instantiated per engine (TC): the SIMT instantiation carries no tensor-core code,
// so the register allocation of its GEMM phase is the one it was tuned with.

// The dynamic shared memory the kernels lay out: for the tensor-core layout its first
// 1024-byte aligned address (128-byte swizzled operands need 1024-byte aligned atoms).
template <typename W>
__device__ __forceinline__ unsigned char* smem_base(unsigned char* raw) {
  if constexpr (kTensorCores<W>) {
    const uint32_t a = smem_u32(raw);
    return raw + ((1024u - (a & 1023u)) & 1023u);
  } else {
    return raw;
  }
}

// Index of decoder pass phase ph among the pass's GEMM phases (6 per layer, then the LM head).
__device__ __forceinline__ int decoder_gemm_index(int ph, int Ld) {
  if (ph == 8 * Ld) return 6 * Ld;
  const int t = ph & 7;
  return 6 * (ph >> 3) + (t == PH_QKV ? TD_QKV : t == PH_O ? TD_O : t == PH_QC ? TD_QC
                          : t == PH_OC ? TD_OC : t == PH_FFN1 ? TD_FFN1 : TD_FFN2);
}

// One GEMM phase; on the tensor-core path a wait that gave up raises the grid's abort flag and
// PD_ETIMEOUT, so the other CTAs leave their next barrier instead of waiting for this one.
template <typename W, bool TC>
__device__ __forceinline__ bool run_gemm(const KParams<W>& P, const GemmArgs<W>& g,
                                         const EmbedTabs<W>& T, int gph, unsigned char* smem) {
  if constexpr (TC) {
    const Dims& D = smem_dims<W>();
    const SmemLayout SL = smem_layout(D, sizeof(W));
    const bool ok = tc_gemm_phase<W>(g, T, D, gph, P.maps, smem + SL.ring, smem + SL.bbuf,
                                     reinterpret_cast<float*>(smem + SL.epi),
                                     reinterpret_cast<Partial*>(smem + SL.scratch), P.B.red,
                                     P.B.cnt);
    if (!ok && threadIdx.x == 0) {
      atomicExch(P.B.bar + 1, 1u);
      atomicCAS(&P.B.st->status, 0, (int)PD_ETIMEOUT);
    }
    return ok;
  } else {
    gemm_phase<W>(g, T, smem_dims<W>(), smem);
    return true;
  }
}

// Thread 0 of a tensor-core kernel: top up the weight stream (while the CTA waits at a grid
// barrier, the slots its last phase used have been released).
template <typename W, bool TC>
__device__ __forceinline__ void stream_weights(const KParams<W>& P, unsigned char* smem) {
  if constexpr (TC) {
    if (threadIdx.x == 0)
      tc_produce<W>(smem_dims<W>(), P.maps,
                    smem + smem_layout(smem_dims<W>(), sizeof(W)).ring, false);
  }
}

// One decoder pass over the M rows described in the commit region, followed by the LM head, as
// a loop over phases separated by grid barriers.  The arguments of the next GEMM phase are
// written to shared memory by one thread while its CTA waits at the barrier, and the weights
// three phases ahead are requested from L2 there, so that neither is on the chain of dependent
// phases.
template <typename W, bool TC>
__device__ bool run_pass(const KParams<W>& P, int M, float* logits, unsigned& tgt,
                         unsigned char* smem, bool pass_open) {
  const Dims& D = smem_dims<W>();
  const Bufs<W>& B = P.B;
  int* status = &B.st->status;
  const SmemLayout SL = smem_layout(D, sizeof(W));
  float* scratch = reinterpret_cast<float*>(smem + SL.scratch);
  const CommitMem cm = commit_mem(D, smem + SL.commit);
  const EmbedTabs<W>& T = smem_tabs<W>();
  GemmArgs<W>& ga = smem_args<W>();
  const int nph = 8 * D.Ld + 1;
  if constexpr (TC) {
    if (threadIdx.x == 0) tc_begin_pass<W>(M, pass_open);
    tc_plan<W>(M);
  }
  if (threadIdx.x == 32) gemm_args(P, 0, M, cm.rtok, cm.rpos, cm.rslot, logits, ga);
  // the SIMT path asks L2 for the weights ahead; the tensor-core path streams them itself (its
  // TMA loads would queue behind bulk L2 prefetches in the same copy engine)
  if constexpr (!TC) prefetch_pass_start(P);
  __syncthreads();
  const size_t self_ld = (size_t)D.kv_pages * kPageRows * D.d;
  const size_t cross_ld = (size_t)D.max_batch * D.max_src * D.d;
  for (int ph = 0; ph < nph; ++ph) {
    const bool attn = is_attn_phase(ph, nph);
    if (attn) {
      const int l = ph >> 3;
      if ((ph & 7) == PH_SELF)
        attn_phase<W, W>(D, B.q, B.kself + l * self_ld, B.vself + l * self_ld, B.att, M,
                         cm.rsb, cm.rkn, 0, scratch, cm.pt);
      else
        attn_phase<W, W>(D, B.q, B.kcross + l * cross_ld, B.vcross + l * cross_ld, B.att, M,
                         cm.rxb, cm.rxn, 0, scratch);
    } else if (!run_gemm<W, TC>(P, ga, T, decoder_gemm_index(ph, D.Ld), smem)) {
      return false;
    }
    if (ph == nph - 1) break;            // the caller's barrier follows the LM head
    const int next = is_attn_phase(ph + 1, nph) ? ph + 2 : ph + 1;
    if (!grid_barrier(B.bar, tgt, status, [&] {
          if (!attn && threadIdx.x == 32)
            gemm_args(P, next, M, cm.rtok, cm.rpos, cm.rslot, logits, ga);
          if constexpr (!TC) prefetch_phase(P, ph + 3);
          stream_weights<W, TC>(P, smem);
        }))
      return false;
  }
  return true;
}

// Shared-memory regions and pass-wide values of the cluster engine's super-phases, kept in
// shared memory (like the GEMM arguments of the SIMT engine) so that the products' loops do
// not hold them in registers.
template <typename W>
struct ClCtx {
  float* ys;
  W* us;
  float* qs;
  W* as;
  W* hs;
  float* red;
  float* sc;
  float* wred;
  int rank, cid, ncl, u, nffn;
  size_t part_ld;
  CommitMem cm;
};
template <typename W>
__device__ __forceinline__ ClCtx<W>& smem_clctx() {
  __shared__ ClCtx<W> s;
  return s;
}
template <typename W>
__device__ __forceinline__ ClGemm<W>& smem_clgemm() {
  __shared__ ClGemm<W> s;
  return s;
}
template <typename W>
__device__ __forceinline__ ClStage<W>& smem_clstage() {
  __shared__ ClStage<W> s;
  return s;
}
// Thread 0, once per kernel.
template <typename W>
__device__ void cl_ctx_init(unsigned char* smem) {
  const Dims& D = smem_dims<W>();
  const SmemLayout SL = smem_layout(D, sizeof(W));
  ClCtx<W>& c = smem_clctx<W>();
  c.ys = reinterpret_cast<float*>(smem + SL.xs);
  c.us = reinterpret_cast<W*>(smem + SL.us);
  c.qs = reinterpret_cast<float*>(smem + SL.qs);
  c.as = reinterpret_cast<W*>(smem + SL.as);
  c.hs = reinterpret_cast<W*>(smem + SL.hs);
  c.red = reinterpret_cast<float*>(smem + SL.part);
  c.sc = reinterpret_cast<float*>(smem + SL.scratch);
  c.wred = c.sc + D.max_keys;
  c.rank = (int)cl_rank();
  c.cid = (int)cl_index();
  c.ncl = (int)cl_count();
  c.u = D.cl_fu * D.cl;
  c.nffn = (D.f + c.u - 1) / c.u;
  c.part_ld = (size_t)D.rows * D.d;
  c.cm = commit_mem(D, smem + SL.commit);
}

// A product of the cluster engine: thread 0 fills the shared argument block (fill(g) on a
// cleared block), the CTA runs it, and meets again before the block can be refilled.
template <typename W, int EPI, bool SHORT = false, typename F>
__device__ __forceinline__ void cl_product(F&& fill) {
  ClGemm<W>& g = smem_clgemm<W>();
  if (threadIdx.x == 0) {
    g = ClGemm<W>{};
    fill(g);
  }
  __syncthreads();
  cl_gemm<W, EPI, SHORT>(g, smem_clctx<W>().red);
  __syncthreads();
}

// Super-phase SA (self) or SB (cross) of layer l for the heads of this cluster: per tile of
// rows, stage, then per head the queries (and self keys / values), attention, and the head's
// share of the output projection into partial sum h of p_out.
template <typename W>
__device__ __noinline__ void cl_attn_super(const KParams<W>& P, int l, bool self, int M,
                                           float* p_out) {
  const Dims& D = smem_dims<W>();
  const ClCtx<W>& c = smem_clctx<W>();
  const int dh = D.dh, cs = D.cl;
  for (int m0 = 0; m0 < M; m0 += kClRows) {
    const int mt = M - m0 < kClRows ? M - m0 : kClRows;
    cl_stage(smem_clstage<W>(), smem_tabs<W>(), D, c.cm.rtok, c.cm.rpos, m0, mt, c.ys, c.us,
             c.red);
    for (int h = c.cid; h < D.H; h += c.ncl) {
      const size_t self_ld = (size_t)D.kv_pages * kPageRows * D.d;
      const size_t cross_ld = (size_t)D.max_batch * D.max_src * D.d;
      // queries (and, self-attention, the keys / values of the tile's rows) of head h
      auto fill_q = [&](ClGemm<W>& g) {
        const DecLayerW<W>& L = smem_mw<W>().dec[l];
        g.m0 = m0; g.mt = mt; g.nct = cs; g.cta = c.rank; g.ncl = cs; g.d = D.d; g.dh = dh;
        g.K = D.d; g.xs = c.us; g.ldx = D.d; g.hoff = h * dh; g.qs = c.qs;
        g.scale = 1.0f / sqrtf((float)dh);
        if (self) {
          g.N = 3 * dh; g.wr = ClRows<W>{L.wqkv, D.d, h * dh, dh, D.d, 0};
          g.epi = CL_QKV; g.bias = L.bqkv; g.slot = c.cm.rslot;
          g.kdst = P.B.kself + l * self_ld; g.vdst = P.B.vself + l * self_ld;
        } else {
          g.N = dh; g.wr = ClRows<W>{L.wqc, D.d, h * dh, dh, 0, 0};
          g.epi = CL_Q; g.bias = L.bqc + h * dh;
        }
      };
      if (self) cl_product<W, CL_QKV>(fill_q);
      else cl_product<W, CL_Q>(fill_q);
      cl_sync();
      // attention of the tile's rows (rows rank, rank + cs, ... of this CTA)
      for (int r = c.rank; r < mt; r += cs) {
        const int m = m0 + r;
        if (self)
          cl_attn_row<W>(D, c.qs + r * dh, P.B.kself + l * self_ld, P.B.vself + l * self_ld,
                         h * dh, c.cm.rkn[m], c.cm.pt, c.cm.rsb[m], c.sc, c.wred, c.as + r * dh);
        else
          cl_attn_row<W>(D, c.qs + r * dh, P.B.kcross + l * cross_ld, P.B.vcross + l * cross_ld,
                         h * dh, c.cm.rxn[m], nullptr, c.cm.rxb[m], c.sc, c.wred, c.as + r * dh);
      }
      cl_sync();
      // head h's share of the output projection: partial sum h
      cl_product<W, CL_PART, true>([&](ClGemm<W>& g) {
        const DecLayerW<W>& L = smem_mw<W>().dec[l];
        g.m0 = m0; g.mt = mt; g.nct = cs; g.cta = c.rank; g.ncl = cs; g.d = D.d; g.dh = dh;
        g.N = D.d; g.K = dh; g.wr = ClRows<W>{self ? L.wo : L.woc, D.d, 0, D.d, 0, h * dh};
        g.xs = c.as; g.ldx = dh; g.epi = CL_PART; g.gout = p_out + (size_t)h * c.part_ld;
      });
    }
  }
}

// Super-phase SC of layer l for this cluster's FFN hidden units: per tile of rows, stage,
// FFN1 of the units with the activation into every CTA's hs, and the units' share of FFN2 into
// partial sum cid of p_out.
template <typename W>
__device__ __noinline__ void cl_ffn_super(const KParams<W>& P, int l, int M, float* p_out) {
  const Dims& D = smem_dims<W>();
  const ClCtx<W>& c = smem_clctx<W>();
  const int cs = D.cl;
  const int c0 = c.cid * c.u, nc = D.f - c0 < c.u ? D.f - c0 : c.u;
  for (int m0 = 0; m0 < M; m0 += kClRows) {
    const int mt = M - m0 < kClRows ? M - m0 : kClRows;
    cl_stage(smem_clstage<W>(), smem_tabs<W>(), D, c.cm.rtok, c.cm.rpos, m0, mt, c.ys, c.us,
             c.red);
    cl_product<W, CL_HID>([&](ClGemm<W>& g) {
      const DecLayerW<W>& L = smem_mw<W>().dec[l];
      g.m0 = m0; g.mt = mt; g.nct = cs; g.cta = c.rank; g.ncl = cs; g.d = D.d;
      g.N = nc; g.K = D.d; g.wr = ClRows<W>{L.w1, D.d, c0, nc, 0, 0}; g.xs = c.us; g.ldx = D.d;
      g.epi = CL_HID; g.bias = L.b1 + c0; g.hs = c.hs; g.ldh = c.u; g.act = D.act;
    });
    cl_sync();
    cl_product<W, CL_PART, true>([&](ClGemm<W>& g) {
      const DecLayerW<W>& L = smem_mw<W>().dec[l];
      g.m0 = m0; g.mt = mt; g.nct = cs; g.cta = c.rank; g.ncl = cs; g.d = D.d;
      g.N = D.d; g.K = nc; g.wr = ClRows<W>{L.w2, D.f, 0, D.d, 0, c0}; g.xs = c.hs; g.ldx = c.u;
      g.epi = CL_PART; g.gout = p_out + (size_t)c.cid * c.part_ld;
    });
  }
}

// The LM head over the whole grid: every cluster stages the final rows for its CTAs; argmax
// partials per CTA and row (or raw logits).
template <typename W>
__device__ __noinline__ void cl_lm_super(const KParams<W>& P, int M, float* logits) {
  const Dims& D = smem_dims<W>();
  const ClCtx<W>& c = smem_clctx<W>();
  for (int m0 = 0; m0 < M; m0 += kClRows) {
    const int mt = M - m0 < kClRows ? M - m0 : kClRows;
    cl_stage(smem_clstage<W>(), smem_tabs<W>(), D, c.cm.rtok, c.cm.rpos, m0, mt, c.ys, c.us,
             c.red);
    auto fill = [&](ClGemm<W>& g) {
      g.m0 = m0; g.mt = mt; g.d = D.d;
      g.N = D.V; g.K = D.d; g.wr = ClRows<W>{smem_mw<W>().embed, D.d, 0, D.V, 0, 0};
      g.xs = c.us; g.ldx = D.d; g.nct = (int)gridDim.x; g.cta = (int)blockIdx.x; g.ncl = D.cl;
      g.epi = logits != nullptr ? CL_LOGITS : CL_ARGMAX;
      g.logits = logits; g.part = P.B.part; g.part_ld = D.rows;
    };
    if (logits != nullptr) cl_product<W, CL_LOGITS>(fill);
    else cl_product<W, CL_ARGMAX>(fill);
  }
}

// Ask L2 for the weight rows this CTA reads in super-phase s (row segments of its product
// groups: group g of a product goes to CTA g mod cs of the cluster), while it waits at the grid
// barrier before it.
template <typename W>
__device__ void cl_prefetch(int s, int tid, int nthreads) {
  const Dims& D = smem_dims<W>();
  const ClCtx<W>& c = smem_clctx<W>();
  if (s >= 3 * D.Ld) return;                     // the LM head's table is asked at pass start
  const int l = s / 3, kind = s - 3 * l, cs = D.cl, dh = D.dh;
  const DecLayerW<W>& L = smem_mw<W>().dec[l];
  // rows of product (wr, N, K) that this CTA's groups read (group g of 4 rows goes to CTA
  // g mod cs), one 16-byte aligned segment each; this thread takes rows tid, tid + nthreads, ...
  // of the CTA's list, numbered on from t
  auto rows = [&](const ClRows<W>& wr, int N, int K, int& t) {
    const int ng = (N + kNCol - 1) / kNCol;
    const int mine = ng > c.rank ? (ng - c.rank + cs - 1) / cs : 0;   // groups of this CTA
    const int nr = mine * kNCol;
    for (int i = ((tid - t) % nthreads + nthreads) % nthreads; i < nr; i += nthreads) {
      const int n = (c.rank + (i / kNCol) * cs) * kNCol + i % kNCol;
      if (n < N) l2_prefetch(wr.row(n), (unsigned)(K * sizeof(W)));
    }
    t += nr;
  };
  int t = 0;
  if (kind < 2) {
    for (int h = c.cid; h < D.H; h += c.ncl) {
      if (kind == 0) rows(ClRows<W>{L.wqkv, D.d, h * dh, dh, D.d, 0}, 3 * dh, D.d, t);
      else rows(ClRows<W>{L.wqc, D.d, h * dh, dh, 0, 0}, dh, D.d, t);
      rows(ClRows<W>{kind == 0 ? L.wo : L.woc, D.d, 0, D.d, 0, h * dh}, D.d, dh, t);
    }
  } else if (c.cid < c.nffn) {
    const int c0 = c.cid * c.u, nc = D.f - c0 < c.u ? D.f - c0 : c.u;
    rows(ClRows<W>{L.w1, D.d, c0, nc, 0, 0}, nc, D.d, t);
    rows(ClRows<W>{L.w2, D.f, 0, D.d, 0, c0}, D.d, nc, t);
  }
}

// One decoder pass of the cluster engine (cl_pass.cuh) over the M rows described in the
// commit region: per layer the super-phases SA (self-attention), SB (cross-attention) and SC
// (FFN), each followed by a grid barrier, then the LM head.  Super-phase s reads the residual
// rows R[s & 1] and the partial sums P[s & 1] the previous one left, and writes R[(s+1) & 1]
// (cluster 0) and P[(s+1) & 1]; the two sets alternate, so no super-phase overwrites what
// another cluster may still be reading.  False if a barrier gave up.
template <typename W>
__device__ bool run_pass_cl(const KParams<W>& P, int M, float* logits, unsigned& tgt,
                            unsigned char* smem) {
  const Dims& D = smem_dims<W>();
  const Bufs<W>& B = P.B;
  const ModelW<W>& mw = smem_mw<W>();
  const bool pre = D.pre_ln != 0;
  const int cid = (int)cl_index();
  const int u = D.cl_fu * D.cl, nffn = (D.f + u - 1) / u;
  const size_t part_ld = (size_t)D.rows * D.d;
  if (threadIdx.x == 0) cl_ctx_init<W>(smem);
  prefetch_gemm_weights(mw.embed, D.V, D.d);       // the LM head's table, asked from L2 early
  __syncthreads();
  cl_prefetch<W>(0, threadIdx.x, blockDim.x);
  for (int s = 0;; ++s) {
    const int l = s / 3, kind = s - 3 * l;        // kind 0 SA, 1 SB, 2 SC; s = 3 Ld: LM head
    const bool lm = s == 3 * D.Ld;
    float* p_out = B.clp + ((s & 1) ? 0 : (size_t)D.cl_np * part_ld);
    if (threadIdx.x == 0) {
      ClStage<W>& st = smem_clstage<W>();
      st = ClStage<W>{};
      st.r_in = (s & 1) ? B.rb : B.ra;
      st.part = B.clp + ((s & 1) ? (size_t)D.cl_np * part_ld : 0);
      st.part_ld = part_ld;
      st.r_out = lm ? nullptr : ((s & 1) ? B.ra : B.rb);
      if (s == 0) {                               // layer 0 starts from the embedding
        st.emb = 1;
        if (pre) { st.lna_g = mw.dec_lne_g; st.lna_b = mw.dec_lne_b; }
      } else {                                    // what the previous super-phase left
        const int pk = (s - 1) % 3;
        const DecLayerW<W>& PL = mw.dec[(s - 1) / 3];
        st.np = pk == 2 ? nffn : D.H;
        st.bias = pk == 0 ? PL.bo : (pk == 1 ? PL.boc : PL.b2);
        if (!pre) {                               // post-LN: the sublayer's LayerNorm
          st.lna_g = pk == 0 ? PL.ln1g : (pk == 1 ? PL.ln2g : PL.ln3g);
          st.lna_b = pk == 0 ? PL.ln1b : (pk == 1 ? PL.ln2b : PL.ln3b);
        }
      }
      if (pre) {                                  // pre-LN: this sublayer's input LayerNorm
        if (lm) {
          st.lnb_g = mw.dec_lnf_g; st.lnb_b = mw.dec_lnf_b;
        } else {
          const DecLayerW<W>& L = mw.dec[l];
          st.lnb_g = kind == 0 ? L.ln1g : (kind == 1 ? L.ln2g : L.ln3g);
          st.lnb_b = kind == 0 ? L.ln1b : (kind == 1 ? L.ln2b : L.ln3b);
        }
      }
    }
    __syncthreads();
    if (lm) {
      cl_lm_super<W>(P, M, logits);
      return true;                                // the caller's barrier follows
    }
    if (kind < 2 && cid < D.H) cl_attn_super<W>(P, l, kind == 0, M, p_out);
    else if (kind == 2 && cid < nffn) cl_ffn_super<W>(P, l, M, p_out);
    if (!cl_grid_barrier(B.bar, tgt, &B.st->status,
                         [&] {               // thread 0 polls: the others ask L2 for weights
                           if (threadIdx.x > 0) cl_prefetch<W>(s + 1, threadIdx.x - 1, blockDim.x - 1);
                         }))
      return false;
  }
}

// ------------------------------------------------------------------------------------------
// fixed-point commit (every CTA): StopC of Eq. 5, block advance of Algorithms 1-3, trace row
// ------------------------------------------------------------------------------------------

// Rows of the next pass: every sentence that is not done contributes its block rows, inputs
// y_{i-1} then the draft at positions i-1..i+blk-2 (the shift-left of Algorithm 2's appendix
// note; under the suffix rule only the rows after the block's exact prefix), sentences in
// order.  All threads of the CTA; misc[0] = the row count.
template <typename W>
__device__ void build_rows(const KParams<W>& P, const CommitMem& cm) {
  const Dims& D = smem_dims<W>();
  const int S = P.n_sent;
  if (threadIdx.x == 0) {
    int r = 0;
    for (int s = 0; s < S; ++s) {
      cm.r0[s] = r;
      if (!cm.st[s].done) r += cm.st[s].blk - cm.st[s].a;
    }
    cm.misc[0] = r;
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // a fresh block's drafts under the last-token rule: y_{i-1} repeated (else they stay PAD)
  for (int s = warp; s < S; s += kWarps) {
    const DecState& st = cm.st[s];
    if (st.done || st.k != 0 || st.init_rule != PD_INIT_LAST || st.method == PD_GREEDY ||
        st.ar_tail)
      continue;
    int* ys = cm.y + (size_t)s * (D.max_tgt + 1);
    const int last = ys[st.i - 1];
    for (int j = lane; j < st.blk; j += 32) ys[st.i + j] = last;
  }
  __syncthreads();
  for (int s = warp; s < S; s += kWarps) {
    const DecState& st = cm.st[s];
    if (st.done) continue;
    const int* ys = cm.y + (size_t)s * (D.max_tgt + 1);
    // rows predict block offsets a..blk-1 (a > 0 only under the suffix rule)
    for (int j = lane; j < st.blk - st.a; j += 32) {
      const int r = cm.r0[s] + j, pos = st.i - 1 + st.a + j;
      cm.rtok[r] = ys[pos];
      cm.rpos[r] = pos;
      cm.rsb[r] = s;
      cm.rslot[r] = page_slot(cm.pt + s * D.pt_ld, pos);
      cm.rkn[r] = pos + 1;                  // block-causal: keys 0..pos of its own sentence
      cm.rxb[r] = s * D.max_src;
      cm.rxn[r] = st.n_src;
    }
  }
  __syncthreads();
}

// Run after the grid barrier that follows the LM head, by every CTA on its own copy of the
// decoding states and of y (shared memory): the CTA partials of each row are merged in the
// same fixed order everywhere, so every CTA takes the same decisions and needs nothing from
// the others.  Thread s decides for sentence s; CTA 0 alone writes the trace (single-sentence
// decodes).  Ends with the rows of the next pass.
template <typename W>
__device__ __noinline__ void commit(const KParams<W>& P, unsigned char* smem) {
  const Dims& D = smem_dims<W>();
  const Bufs<W>& B = P.B;
  const SmemLayout SL = smem_layout(D, sizeof(W));
  const CommitMem cm = commit_mem(D, smem + SL.commit);
  const int tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;
  const int M = cm.misc[0], S = P.n_sent;
  // per row: the CTA partials merged lane-wise in ascending CTA order (loads issued in
  // batches), then by a fixed butterfly (the merge is symmetric, so every lane ends with the
  // same result); a NaN row gets token -1
  constexpr int kBatch = 8;
  for (int r = warp; r < M; r += kWarps) {
    Partial a{-INFINITY, 0x7fffffff, 0.f, 0};
    for (int c0 = 0; c0 < (int)gridDim.x; c0 += 32 * kBatch) {
      Partial v[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int c = c0 + 32 * j + lane;
        if (c < (int)gridDim.x) v[j] = B.part[(size_t)c * D.rows + r];
      }
#pragma unroll
      for (int j = 0; j < kBatch; ++j)
        if (c0 + 32 * j + lane < (int)gridDim.x) partial_merge(a, v[j]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const Partial b = shfl_partial(a, o);
      partial_merge(a, b);
    }
    if (lane == 0) {
      cm.ntok[r] = (a.nan || a.mx == -INFINITY) ? -1 : a.idx;
      cm.nprob[r] = 1.0f / a.sum;
    }
  }
  __syncthreads();
  for (int s = tid; s < S; s += blockDim.x) {
    DecState st = cm.st[s];                        // decisions on a register copy
    if (st.done) continue;
    const int r0 = cm.r0[s], blk = st.blk, i = st.i, a = st.a;
    const int* nt = cm.ntok + r0 - a;              // the pass's rows are block offsets a..blk-1
    const int* ys = cm.y + (size_t)s * (D.max_tgt + 1);
    // the block's new tokens: offsets below a were exact before this pass and stay as they are
    auto newtok = [&](int off) { return off < a ? ys[i + off] : nt[off]; };
    bool nan = false;
    for (int r = a; r < blk; ++r) nan = nan || nt[r] < 0;
    int c = a;                                     // leading positions equal to the old draft
    while (c < blk && nt[c] == ys[i + c]) ++c;
    const int stop = c == blk;
    int eos_idx = -1;
    for (int r = 0; r < blk; ++r)
      if (newtok(r) == D.eos) { eos_idx = r; break; }
    st.k = st.k + 1;
    const int n_it = st.n_iters + 1;
    st.n_iters = n_it;
    const int t = st.n_trace;
    if (t < D.max_tgt) {
      if (S == 1 && blockIdx.x == 0) {
        pd_trace_step row;
        row.step = n_it; row.block_start = i; row.block_len = blk; row.n_converged = c;
        row.stop = stop; row.eos_idx = eos_idx; row.n_rows = blk - a;
        B.trace[t] = row;
        for (int r = 0; r < blk; ++r) {
          B.trace_tok[(size_t)t * D.max_tgt + r] = newtok(r);
          // a row not re-run keeps the probability of the pass that made it exact
          B.trace_prob[(size_t)t * D.max_tgt + r] =
              r < a ? B.trace_prob[(size_t)(t - 1) * D.max_tgt + r] : cm.nprob[r0 + r - a];
        }
      }
      st.n_trace = t + 1;
    }
    if (nan) {
      st.status = PD_ENAN; st.n_y = i - 1; st.done = 1;
    } else {
      // the block is solved: StopC, the pass cap, or (accepted-prefix and suffix rules) the
      // first c + 1 new tokens exact with c + 1 >= blk
      const bool prefix = st.stop_rule == PD_STOP_PREFIX || st.stop_rule == PD_STOP_SUFFIX;
      if (stop || st.k >= blk || (prefix && c + 1 >= blk)) {
        st.a = 0;
        const bool one_pos = st.method == PD_GREEDY || st.ar_tail;
        if (one_pos) {
          const bool eos_ends = st.ar_tail ? true : (st.stop_at_eos != 0);
          if (eos_ends && newtok(0) == D.eos) { st.n_y = i; st.done = 1; }
        } else if (st.method == PD_HYBRID_GS_JACOBI && eos_idx >= 0) {
          st.n_y = i + eos_idx;                    // through the EOS (Algorithm 3)
          st.done = 1;
        }
        if (!st.done) {
          const int ni = i + blk;
          if (st.method == PD_HYBRID_GS_JACOBI && !st.ar_tail && ni > st.h) {
            st.ar_tail = 1;                        // greedy tail up to max_len
            st.b_eff = 1;
            st.m_eff = st.max_len;
          }
          if (ni > st.m_eff) {
            st.done = 1;
            st.n_y = st.m_eff;
            st.scan = (st.method == PD_JACOBI || st.method == PD_GS_JACOBI) && st.stop_at_eos;
          } else {
            st.i = ni;
            const int rest = st.m_eff - ni + 1;
            st.blk = st.b_eff < rest ? st.b_eff : rest;
            st.k = 0;
          }
        }
      } else if (st.stop_rule == PD_STOP_SUFFIX) {
        st.a = c + 1;                              // the next pass re-runs offsets c+1..blk-1
      }
      // the pass budget, and a hard cap no correct schedule reaches (at most m passes for the
      // parallel part plus max_len for a greedy tail): the loop can never run away
      if (!st.done && ((st.max_passes > 0 && n_it >= st.max_passes) || n_it > 2 * st.max_len + 2)) {
        st.status = PD_ENOTCONV;
        st.n_y = st.i - 1;
        st.done = 1;
      }
    }
    cm.st[s] = st;
  }
  __syncthreads();
  for (int r = tid; r < M; r += blockDim.x)        // y_{i:i+blk} <- new, every sentence
    cm.y[(size_t)cm.rsb[r] * (D.max_tgt + 1) + cm.rpos[r] + 1] = cm.ntok[r];
  __syncthreads();
  for (int s = tid; s < S; s += blockDim.x) {      // the first EOS among y_1..y_m ends y
    DecState& st = cm.st[s];
    if (!st.scan) continue;
    const int* ys = cm.y + (size_t)s * (D.max_tgt + 1);
    for (int p = 1; p <= st.m_eff; ++p)
      if (ys[p] == D.eos) { st.n_y = p; break; }
    st.scan = 0;
  }
  __syncthreads();
  build_rows(P, cm);
}

// CTA 0, at the end of a decode: tokens and info of every sentence from its copies of the
// states; a failure a device-side wait recorded in the status word (PD_ETIMEOUT) takes
// precedence.
template <typename W>
__device__ void write_outputs(const KParams<W>& P, unsigned char* smem) {
  const Dims& D = smem_dims<W>();
  const SmemLayout SL = smem_layout(D, sizeof(W));
  const CommitMem cm = commit_mem(D, smem + SL.commit);
  const int S = P.n_sent;
  __syncthreads();
  if (P.out_info == nullptr) return;
  for (int s = 0; s < S; ++s) {
    const int n_y = cm.st[s].n_y;
    const int* ys = cm.y + (size_t)s * (D.max_tgt + 1);
    for (int p = threadIdx.x; p < n_y; p += blockDim.x) P.out_y[(size_t)s * P.out_ld + p] = ys[1 + p];
  }
  if (threadIdx.x == 0) {
    const int g = atomicAdd(&P.B.st->status, 0);
    for (int s = 0; s < S; ++s) {
      const DecState& st = cm.st[s];
      P.out_info[4 * s + 0] = st.n_y;
      P.out_info[4 * s + 1] = st.n_iters;
      P.out_info[4 * s + 2] = g != 0 ? g : st.status;
      P.out_info[4 * s + 3] = st.n_trace;
    }
  }
}

// ------------------------------------------------------------------------------------------
// kernels
// ------------------------------------------------------------------------------------------

template <typename W, bool TC, bool CL = false>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const __grid_constant__ KParams<W> P) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  unsigned char* smem = smem_base<W>(smem_raw);
  unsigned tgt = 0;
  const Dims& D = smem_dims<W>();
  const Bufs<W>& B = P.B;
  int* status = &B.st->status;
  load_smem_mw(P);
  load_smem_vectors<W>(D, smem);
  const SmemLayout SL = smem_layout(D, sizeof(W));
  const CommitMem cm = commit_mem(D, smem + SL.commit);
  if constexpr (TC) tc_setup<W>(D, TC_DECODE, SL.ring_slots, P.maps);

  for (int e = threadIdx.x; e < D.max_batch * D.pt_ld; e += blockDim.x) cm.pt[e] = B.page_tab[e];
  __syncthreads();

  if (P.debug_len > 0) {                  // teacher-forced rows 0..len-1 of the slot-0 sentence
    for (int m = threadIdx.x; m < P.debug_len; m += blockDim.x) {
      cm.rtok[m] = B.dbg_tok[m];
      cm.rpos[m] = m; cm.rslot[m] = page_slot(cm.pt, m); cm.rsb[m] = 0; cm.rkn[m] = m + 1;
      cm.rxb[m] = 0; cm.rxn[m] = P.n_src_s[0];
    }
    __syncthreads();
    if constexpr (CL) {
      run_pass_cl<W>(P, P.debug_len, P.logits, tgt, smem);
      cl_sync();                          // no CTA leaves while a partner may read its memory
    } else {
      run_pass<W, TC>(P, P.debug_len, P.logits, tgt, smem, false);
    }
    if constexpr (TC) tc_teardown<W>();
    return;
  }

  // every CTA: its copies of the states and of y_0..y_m; InitT = all PAD (Section 3.3)
  const int S = P.n_sent;
  for (int s = threadIdx.x; s < S; s += blockDim.x) {
    DecState st = P.init;
    st.max_len = P.max_len_s[s];
    st.h = (P.init.h <= 0 || P.init.h > st.max_len) ? st.max_len : P.init.h;
    st.n_src = P.n_src_s[s];
    st.b_eff = st.method == PD_GREEDY ? 1 : (st.method == PD_JACOBI ? st.max_len : st.b);
    st.m_eff = st.method == PD_HYBRID_GS_JACOBI ? st.h : st.max_len;
    st.i = 1;
    st.blk = st.b_eff < st.m_eff ? st.b_eff : st.m_eff;
    st.k = 0; st.ar_tail = 0; st.n_iters = 0; st.done = 0; st.n_y = 0; st.n_trace = 0;
    st.status = 0; st.scan = 0; st.a = 0;
    cm.st[s] = st;
  }
  for (int e = threadIdx.x; e < S * (D.max_tgt + 1); e += blockDim.x)
    cm.y[e] = e % (D.max_tgt + 1) == 0 ? D.bos : D.pad;
  if (blockIdx.x == 0 && threadIdx.x == 0) *status = 0;   // read by no one before a wait
  __syncthreads();
  build_rows(P, cm);

  for (;;) {
    const int M = cm.misc[0];
    if (M == 0) break;
    if constexpr (CL) {
      if (!run_pass_cl<W>(P, M, nullptr, tgt, smem)) break;
      if (!cl_grid_barrier(B.bar, tgt, status)) break;
    } else {
      if (!run_pass<W, TC>(P, M, nullptr, tgt, smem, true)) break;
      if (!grid_barrier(B.bar, tgt, status, [&] { stream_weights<W, TC>(P, smem); })) break;
    }
    commit<W>(P, smem);
  }
  if (blockIdx.x == 0) write_outputs(P, smem);
  if constexpr (TC) tc_teardown<W>();
  if constexpr (CL) cl_sync();
}

// The encoder pass of encode_kernel: every encoder layer (QKV, full self-attention, O, FFN1,
// FFN2, phases separated by grid barriers), then the cross-attention keys and values of every
// decoder layer from the encoder output.  False if a barrier or a wait gave up.
template <typename W, bool TC>
__device__ bool encode_pass(const KParams<W>& P, unsigned char* smem, unsigned& tgt) {
  const Dims& D = smem_dims<W>();
  const Bufs<W>& B = P.B;
  const ModelW<W>& mw = smem_mw<W>();
  int* status = &B.st->status;
  const SmemLayout SL = smem_layout(D, sizeof(W));
  float* scratch = reinterpret_cast<float*>(smem + SL.scratch);
  const EmbedTabs<W>& T = smem_tabs<W>();
  const bool pre = D.pre_ln != 0;
  const int n = P.n_src;
  const CommitMem cm = commit_mem(D, smem + SL.commit);
  for (int m = threadIdx.x; m < n; m += blockDim.x) cm.rpos[m] = m;   // source positions
  if constexpr (TC) {
    if (threadIdx.x == 0) tc_begin_pass<W>(n, false);
    tc_plan<W>(n);
  }
  __syncthreads();

  if constexpr (!TC) {
    for (int l = 0; l < D.Le; ++l) {
      const EncLayerW<W>& L = mw.enc[l];
      prefetch_gemm_weights(L.wqkv, 3 * D.d, D.d);
      prefetch_gemm_weights(L.wo, D.d, D.d);
      prefetch_gemm_weights(L.w1, D.f, D.d);
      prefetch_gemm_weights(L.w2, D.d, D.f);
    }
    for (int l = 0; l < D.Ld; ++l) prefetch_gemm_weights(mw.dec[l].wkvc, 2 * D.d, D.d);
  }
  auto barrier = [&] { return grid_barrier(B.bar, tgt, status, [&] { stream_weights<W, TC>(P, smem); }); };

  for (int l = 0; l < D.Le; ++l) {
    const EncLayerW<W>& L = mw.enc[l];
    GemmArgs<W> g{};
    g.M = n; g.N = 3 * D.d; g.K = D.d;
    if (l == 0) {
      g.emb_tok = P.enc_tok; g.emb_pos = cm.rpos; g.x_store = B.ra;   // positions 0..n-1
      if (pre) { g.ln_a_g = mw.enc_lne_g; g.ln_a_b = mw.enc_lne_b; g.ln_b_g = L.ln1g; g.ln_b_b = L.ln1b; }
    } else {
      g.x_src = B.ra;
      if (pre) { g.ln_b_g = L.ln1g; g.ln_b_b = L.ln1b; }
      else { g.ln_a_g = mw.enc[l - 1].ln2g; g.ln_a_b = mw.enc[l - 1].ln2b; g.x_store = B.xa; }
    }
    const float* res1 = (pre || l == 0) ? B.ra : B.xa;
    g.w = L.wqkv; g.bias = L.bqkv; g.epi = EPI_QKV; g.out = B.q; g.ld = D.d;
    g.kdst_f = B.k; g.vdst_f = B.v;
    gemm_plan(g, gridDim.x);
    if (!run_gemm<W, TC>(P, g, T, 4 * l + TE_QKV, smem) || !barrier()) return false;

    attn_phase<float, W>(D, B.q, B.k, B.v, B.att, n, nullptr, nullptr, n, scratch);
    if (!barrier()) return false;

    g = GemmArgs<W>{};
    g.M = n; g.N = D.d; g.K = D.d; g.xw_src = B.att; g.w = L.wo; g.bias = L.bo;
    g.epi = EPI_RESID; g.out = B.rb; g.ld = D.d; g.resid = res1;
    gemm_plan(g, gridDim.x);
    if (!run_gemm<W, TC>(P, g, T, 4 * l + TE_O, smem) || !barrier()) return false;

    g = GemmArgs<W>{};
    g.M = n; g.N = D.f; g.K = D.d; g.x_src = B.rb;
    if (pre) { g.ln_b_g = L.ln2g; g.ln_b_b = L.ln2b; }
    else { g.ln_a_g = L.ln1g; g.ln_a_b = L.ln1b; g.x_store = B.xb; }
    const float* res2 = pre ? B.rb : B.xb;
    g.w = L.w1; g.bias = L.b1; g.epi = EPI_ACT; g.out_w = B.ffh; g.ld = D.f;
    gemm_plan(g, gridDim.x);
    if (!run_gemm<W, TC>(P, g, T, 4 * l + TE_FFN1, smem) || !barrier()) return false;

    g = GemmArgs<W>{};
    g.M = n; g.N = D.d; g.K = D.f; g.xw_src = B.ffh; g.w = L.w2; g.bias = L.b2;
    g.epi = EPI_RESID; g.out = B.ra; g.ld = D.d; g.resid = res2;
    gemm_plan(g, gridDim.x);
    if (!run_gemm<W, TC>(P, g, T, 4 * l + TE_FFN2, smem) || !barrier()) return false;
  }
  // cross-attention keys and values of every decoder layer from the encoder output, into the
  // sentence's slot (independent phases: no barrier between them, unless their K is split,
  // whose partial sums and arrival counters the next phase reuses)
  const size_t cross_ld = (size_t)D.max_batch * D.max_src * D.d;
  const size_t slot_off = (size_t)P.enc_slot * D.max_src * D.d;
  for (int l = 0; l < D.Ld; ++l) {
    GemmArgs<W> g{};
    g.M = n; g.N = 2 * D.d; g.K = D.d; g.x_src = B.ra;
    g.ln_b_g = pre ? mw.enc_lnf_g : mw.enc[D.Le - 1].ln2g;
    g.ln_b_b = pre ? mw.enc_lnf_b : mw.enc[D.Le - 1].ln2b;
    g.w = mw.dec[l].wkvc; g.bias = mw.dec[l].bkvc; g.epi = EPI_KVCROSS;
    g.kdst = B.kcross + l * cross_ld + slot_off;
    g.vdst = B.vcross + l * cross_ld + slot_off;
    gemm_plan(g, gridDim.x);
    if (!run_gemm<W, TC>(P, g, T, 4 * D.Le + l, smem)) return false;
    if constexpr (TC) {
      if (l + 1 < D.Ld && gemm_geom(D, TC_ENCODE, 4 * D.Le + l).S > 1 && !barrier()) return false;
    }
  }
  return true;
}

template <typename W, bool TC>
__global__ void __launch_bounds__(kThreads, 1) encode_kernel(const __grid_constant__ KParams<W> P) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  unsigned char* smem = smem_base<W>(smem_raw);
  unsigned tgt = 0;
  load_smem_mw(P);
  const Dims& D = smem_dims<W>();
  if constexpr (TC) tc_setup<W>(D, TC_ENCODE, smem_layout(D, sizeof(W)).ring_slots, P.maps);
  (void)encode_pass<W, TC>(P, smem, tgt);
  if constexpr (TC) tc_teardown<W>();
}

}  // namespace pd


// ============================================================================================
// host side
// ============================================================================================

using pd::Dims;

struct pd_ctx {
  pd_config cfg;
  Dims D;
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  int device = 0, n_sm = 0, grid = 0;
  int cl_grid = 0;                            // cluster engine: CTAs of the decode grid
  size_t smem = 0;
  std::vector<void*> allocs;
  void* wdev = nullptr;                       // device weights (tensors 256-byte aligned)
  std::vector<size_t> woff, wbytes;           // per tensor, blob order
  size_t blob_bytes = 0;
  void* mw_dev = nullptr;                     // ModelW<W> table on the device
  pd::Bufs<float> bf{};
  pd::Bufs<__nv_bfloat16> bb{};
  int32_t* d_out_y = nullptr;
  int32_t* d_out_info = nullptr;
  int n_src_slot[pd::kMaxBatch] = {};        // source length encoded into each cache slot
  int n_encoded = 0;                          // slots 0..n_encoded-1 hold encoded sentences
  int64_t launches = 0;
  float* static_logits = nullptr;              // device address of the fixed logits array
  std::vector<CUtensorMap> dec_maps, enc_maps; // bf16: per GEMM phase of each kernel
  std::vector<int32_t> page_host;              // the sentences' page tables of the last decode
  std::string err;
};

namespace {

pd_status fail(pd_ctx* c, pd_status s, const std::string& msg) {
  if (c) c->err = msg;
  return s;
}

#define PD_CUDA(ctx, call)                                                             \
  do {                                                                                 \
    cudaError_t e_ = (call);                                                           \
    if (e_ != cudaSuccess)                                                             \
      return fail(ctx, PD_ECUDA, std::string(#call ": ") + cudaGetErrorString(e_));    \
  } while (0)

size_t wsize(const pd_config& c) { return c.dtype == PD_DTYPE_BF16 ? 2 : 4; }

bool valid_config(const pd_config* c, std::string* why) {
  auto bad = [&](const char* m) { if (why) *why = m; return false; };
  if (!c) return bad("cfg is NULL");
  if (c->dtype != PD_DTYPE_F32 && c->dtype != PD_DTYPE_BF16) return bad("dtype");
  if (c->d_model <= 0 || c->d_model % 256 || c->d_model > 1024)
    return bad("d_model must be 256, 512, 768 or 1024");
  if (c->d_ff <= 0 || c->d_ff % 256) return bad("d_ff must be a positive multiple of 256");
  if (c->n_heads <= 0 || c->d_model % c->n_heads) return bad("n_heads must divide d_model");
  const int dh = c->d_model / c->n_heads;
  if (dh != 32 && dh != 64 && dh != 128) return bad("d_model / n_heads must be 32, 64 or 128");
  if (c->n_enc_layers < 1 || c->n_enc_layers > pd::kMaxLayers) return bad("n_enc_layers");
  if (c->n_dec_layers < 1 || c->n_dec_layers > pd::kMaxLayers) return bad("n_dec_layers");
  if (c->vocab < 4) return bad("vocab");
  if (c->activation < 0 || c->activation > 2) return bad("activation");
  if (c->learned_pos && c->max_pos < 1) return bad("max_pos");
  if (c->max_src_len < 1 || c->max_tgt_len < 1 || c->max_src_len > 4096 || c->max_tgt_len > 4096)
    return bad("max_src_len / max_tgt_len must be in [1, 4096]");
  for (int id : {c->pad_id, c->eos_id, c->bos_id})
    if (id < 0 || id >= c->vocab) return bad("special ids must be in [0, vocab)");
  if (!(c->ln_eps >= 0.f)) return bad("ln_eps");
  if (c->max_batch < 0 || c->max_batch > pd::kMaxBatch) return bad("max_batch must be in [0, 64]");
  if (c->gemm_engine < PD_ENGINE_AUTO || c->gemm_engine > PD_ENGINE_CLUSTER) return bad("gemm_engine");
  if (c->gemm_engine == PD_ENGINE_TENSOR && c->dtype != PD_DTYPE_BF16)
    return bad("the tensor-core engine needs bf16 weights");
  if (c->cluster_size != 0 && c->cluster_size != 1 && c->cluster_size != 2 &&
      c->cluster_size != 4 && c->cluster_size != 8)
    return bad("cluster_size must be 0, 1, 2, 4 or 8");
  if (c->kv_pages != 0 &&
      (c->kv_pages < (c->max_tgt_len + pd::kPageRows - 1) / pd::kPageRows || c->kv_pages > (1 << 20)))
    return bad("kv_pages must be 0 or hold one sentence of max_tgt_len (<= 2^20 pages)");
  if (c->dtype == PD_DTYPE_BF16 && c->vocab < pd::kTileN)
    return bad("bf16 models need vocab >= 128 (one tensor-core tile)");
  return true;
}

// Tensor sizes (elements) in blob order; the same order fills the pointer table.
template <typename W>
std::vector<std::pair<const W**, size_t>> layout(pd::ModelW<W>& mw, const pd_config& c) {
  const size_t d = c.d_model, f = c.d_ff, V = c.vocab;
  std::vector<std::pair<const W**, size_t>> t;
  t.push_back({&mw.embed, V * d});
  if (c.learned_pos) t.push_back({&mw.pos, (size_t)c.max_pos * d});
  if (c.pre_ln) {
    t.push_back({&mw.enc_lne_g, d}); t.push_back({&mw.enc_lne_b, d});
    t.push_back({&mw.dec_lne_g, d}); t.push_back({&mw.dec_lne_b, d});
    t.push_back({&mw.enc_lnf_g, d}); t.push_back({&mw.enc_lnf_b, d});
    t.push_back({&mw.dec_lnf_g, d}); t.push_back({&mw.dec_lnf_b, d});
  }
  for (int l = 0; l < c.n_enc_layers; ++l) {
    auto& L = mw.enc[l];
    t.push_back({&L.wqkv, 3 * d * d}); t.push_back({&L.bqkv, 3 * d});
    t.push_back({&L.wo, d * d}); t.push_back({&L.bo, d});
    t.push_back({&L.ln1g, d}); t.push_back({&L.ln1b, d});
    t.push_back({&L.w1, f * d}); t.push_back({&L.b1, f});
    t.push_back({&L.w2, d * f}); t.push_back({&L.b2, d});
    t.push_back({&L.ln2g, d}); t.push_back({&L.ln2b, d});
  }
  for (int l = 0; l < c.n_dec_layers; ++l) {
    auto& L = mw.dec[l];
    t.push_back({&L.wqkv, 3 * d * d}); t.push_back({&L.bqkv, 3 * d});
    t.push_back({&L.wo, d * d}); t.push_back({&L.bo, d});
    t.push_back({&L.ln1g, d}); t.push_back({&L.ln1b, d});
    t.push_back({&L.wqc, d * d}); t.push_back({&L.bqc, d});
    t.push_back({&L.wkvc, 2 * d * d}); t.push_back({&L.bkvc, 2 * d});
    t.push_back({&L.woc, d * d}); t.push_back({&L.boc, d});
    t.push_back({&L.ln2g, d}); t.push_back({&L.ln2b, d});
    t.push_back({&L.w1, f * d}); t.push_back({&L.b1, f});
    t.push_back({&L.w2, d * f}); t.push_back({&L.b2, d});
    t.push_back({&L.ln3g, d}); t.push_back({&L.ln3b, d});
  }
  return t;
}

// 1: the tensor is a LayerNorm gain, 2: a LayerNorm bias, 0: a weight or a linear bias.
template <typename W>
int ln_kind(const pd::ModelW<W>& mw, const W** field) {
  const W* const* gains[] = {&mw.enc_lne_g, &mw.dec_lne_g, &mw.enc_lnf_g, &mw.dec_lnf_g};
  const W* const* biases[] = {&mw.enc_lne_b, &mw.dec_lne_b, &mw.enc_lnf_b, &mw.dec_lnf_b};
  for (auto g : gains) if (g == field) return 1;
  for (auto b : biases) if (b == field) return 2;
  for (int l = 0; l < pd::kMaxLayers; ++l) {
    const auto& E = mw.enc[l];
    const auto& L = mw.dec[l];
    if (field == &E.ln1g || field == &E.ln2g || field == &L.ln1g || field == &L.ln2g ||
        field == &L.ln3g)
      return 1;
    if (field == &E.ln1b || field == &E.ln2b || field == &L.ln1b || field == &L.ln2b ||
        field == &L.ln3b)
      return 2;
  }
  return 0;
}

size_t blob_elems(const pd_config& c) {
  pd::ModelW<float> mw{};
  size_t n = 0;
  for (auto& e : layout<float>(mw, c)) n += e.second;
  return n;
}

template <typename W>
pd::Bufs<W>& bufs(pd_ctx* c);
template <> pd::Bufs<float>& bufs<float>(pd_ctx* c) { return c->bf; }
template <> pd::Bufs<__nv_bfloat16>& bufs<__nv_bfloat16>(pd_ctx* c) { return c->bb; }

template <typename T>
pd_status dalloc(pd_ctx* c, T** p, size_t count) {
  void* q = nullptr;
  cudaError_t e = cudaMalloc(&q, count * sizeof(T) > 0 ? count * sizeof(T) : 16);
  if (e != cudaSuccess) return fail(c, PD_ENOMEM, std::string("cudaMalloc: ") + cudaGetErrorString(e));
  c->allocs.push_back(q);
  *p = static_cast<T*>(q);
  return PD_OK;
}

#define PD_TRY(expr)               \
  do {                             \
    pd_status s_ = (expr);         \
    if (s_ != PD_OK) return s_;    \
  } while (0)

// The decode / encode kernel of a context's engine (bf16 only has the tensor-core one; the
// cluster engine's encoder is the SIMT one).
template <typename W>
const void* kernel_fn(bool encode, bool tc, bool cl = false) {
  if constexpr (sizeof(W) == 2) {
    if (tc) return encode ? (const void*)pd::encode_kernel<W, true>
                          : (const void*)pd::decode_kernel<W, true>;
  }
  if (cl && !encode) return (const void*)pd::decode_kernel<W, false, true>;
  return encode ? (const void*)pd::encode_kernel<W, false> : (const void*)pd::decode_kernel<W, false>;
}

pd_status raise_smem_limit(pd_ctx* c, const void* fn) {
  cudaFuncAttributes a{};
  PD_CUDA(c, cudaFuncGetAttributes(&a, fn));
  if ((size_t)a.maxDynamicSharedSizeBytes < c->smem)
    PD_CUDA(c, cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)c->smem));
  return PD_OK;
}

// cuTensorMapEncodeTiled from the driver (through the runtime's entry-point query, so the
// library needs no link against the driver library).
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Tensor-core resources of a bf16 context: a TMA tensor map per weight matrix ([N][K] bf16,
// boxes of 128 rows x 64 K elements with the 128-byte swizzle the MMA's shared-memory
// descriptors expect; rows past N read as zero), the split-K partial buffer and its arrival
// counters.
pd_status tc_resources(pd_ctx* c, const pd::ModelW<__nv_bfloat16>& mw) {
  const Dims& D = c->D;
  PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (!enc) return fail(c, PD_ECUDA, "cuTensorMapEncodeTiled is not available from the driver");
  auto make = [&](CUtensorMap* m, const __nv_bfloat16* w, int N, int K) -> pd_status {
    std::memset(m, 0, sizeof(CUtensorMap));
    cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)N};
    cuuint64_t strides[1] = {(cuuint64_t)K * 2};
    cuuint32_t box[2] = {(cuuint32_t)pd::kKBlock, (cuuint32_t)pd::kTileN};
    cuuint32_t estr[2] = {1, 1};
    const CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<__nv_bfloat16*>(w),
                           dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                           CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(c, PD_ECUDA, "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")");
    return PD_OK;
  };
  // the weight matrix of GEMM phase g of each kernel's phase sequence (pd::gemm_geom order)
  for (int kind : {pd::TC_DECODE, pd::TC_ENCODE}) {
    std::vector<CUtensorMap>& maps = kind == pd::TC_DECODE ? c->dec_maps : c->enc_maps;
    const int n = pd::gemm_phase_count(D, kind);
    maps.assign(n, CUtensorMap{});
    for (int g = 0; g < n; ++g) {
      const pd::Geom G = pd::gemm_geom(D, kind, g);
      const __nv_bfloat16* w;
      if (kind == pd::TC_DECODE) {
        if (g == 6 * D.Ld) {
          w = mw.embed;
        } else {
          const auto& L = mw.dec[g / 6];
          const __nv_bfloat16* t[6] = {L.wqkv, L.wo, L.wqc, L.woc, L.w1, L.w2};
          w = t[g % 6];
        }
      } else if (g >= 4 * D.Le) {
        w = mw.dec[g - 4 * D.Le].wkvc;
      } else {
        const auto& L = mw.enc[g / 4];
        const __nv_bfloat16* t[4] = {L.wqkv, L.wo, L.w1, L.w2};
        w = t[g % 4];
      }
      PD_TRY(make(&maps[g], w, G.N, G.K));
    }
  }
  // the largest split-K partial buffer any GEMM phase needs: S x N x rows floats
  size_t red = 1;
  for (int kind : {pd::TC_DECODE, pd::TC_ENCODE})
    for (int g = 0; g < pd::gemm_phase_count(D, kind); ++g) {
      const pd::Geom G = pd::gemm_geom(D, kind, g);
      if (G.S > 1) red = std::max(red, (size_t)G.S * G.N * D.rows);
    }
  pd::Bufs<__nv_bfloat16>& B = c->bb;
  PD_TRY(dalloc(c, &B.red, red));
  PD_TRY(dalloc(c, &B.cnt, (size_t)pd::kCounterSlots));
  PD_CUDA(c, cudaMemset(B.cnt, 0, pd::kCounterSlots * sizeof(unsigned)));
  return PD_OK;
}

// Cluster-engine geometry of a context: as many clusters of D.cl CTAs as can be resident at
// once with the decode kernel's shared memory (at most n_sm / D.cl), FFN hidden units per CTA
// so that the clusters cover d_ff, and the partial-sum buffers ([2][max(H, FFN slices)][rows]
// [d] fp32).  The FFN share and the shared memory depend on each other, so the two are
// settled together.
template <typename W>
pd_status cl_resources(pd_ctx* c) {
  Dims& D = c->D;
  const void* fdec = kernel_fn<W>(false, false, true);
  Dims De = D;
  De.cl = 0;
  const size_t smem_enc = pd::smem_layout(De, sizeof(W)).total;   // the (SIMT) encoder's
  int ncl = c->n_sm / D.cl;
  for (int it = 0;; ++it) {
    D.cl_n = ncl;
    // units per cluster: a multiple of 16, so that every slice starts on a 16-byte boundary
    // of the FFN2 rows and holds whole 16-byte chunks
    const int per = (D.f + ncl - 1) / ncl, u = (per + 15) / 16 * 16, nffn = (D.f + u - 1) / u;
    D.cl_fu = u / D.cl;
    D.cl_np = std::max(D.H, nffn);
    const size_t smem = std::max(pd::smem_layout(D, sizeof(W)).total, smem_enc);
    if (smem > pd::kSmemMax)
      return fail(c, PD_EINVAL, "the cluster engine's shared memory does not fit (max_tgt_len "
                                "or max_batch too large)");
    cudaFuncAttributes a{};
    PD_CUDA(c, cudaFuncGetAttributes(&a, fdec));
    if ((size_t)a.maxDynamicSharedSizeBytes < smem)
      PD_CUDA(c, cudaFuncSetAttribute(fdec, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    cudaLaunchConfig_t lc{};
    lc.gridDim = dim3(ncl * D.cl);
    lc.blockDim = dim3(pd::kThreads);
    lc.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = (unsigned)D.cl;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.attrs = at;
    lc.numAttrs = 1;
    int fit = 0;
    PD_CUDA(c, cudaOccupancyMaxActiveClusters(&fit, fdec, &lc));
    if (fit >= ncl) break;
    if (fit < 1 || it >= 8) return fail(c, PD_EINVAL, "no cluster of the decode kernel fits an SM group");
    ncl = fit;
  }
  c->cl_grid = D.cl_n * D.cl;
  pd::Bufs<W>& B = bufs<W>(c);
  PD_TRY(dalloc(c, &B.clp, 2 * (size_t)D.cl_np * D.rows * D.d));
  return PD_OK;
}

template <typename W>
pd_status create_impl(pd_ctx* c, const void* weights) {
  const pd_config& cfg = c->cfg;
  Dims& D = c->D;
  // weights: each tensor at a 256-byte aligned offset of one allocation
  pd::ModelW<W> mw{};
  auto lay = layout<W>(mw, cfg);
  size_t off = 0;
  for (auto& e : lay) {
    c->woff.push_back(off);
    c->wbytes.push_back(e.second * sizeof(W));
    off += (e.second * sizeof(W) + 255) / 256 * 256;
  }
  unsigned char* wdev = nullptr;
  PD_TRY(dalloc(c, &wdev, off));
  c->wdev = wdev;
  const unsigned char* src = static_cast<const unsigned char*>(weights);
  size_t soff = 0;
  for (size_t k = 0; k < lay.size(); ++k) {
    *lay[k].first = reinterpret_cast<const W*>(wdev + c->woff[k]);
    if (src != nullptr) {
      PD_CUDA(c, cudaMemcpy(wdev + c->woff[k], src + soff, c->wbytes[k], cudaMemcpyHostToDevice));
    } else {                             // no blob: draw the weights from cfg.seed
      pd::seeded_weights_kernel<W><<<c->n_sm * 4, 256, 0, c->stream>>>(
          reinterpret_cast<W*>(wdev + c->woff[k]), lay[k].second, (unsigned)k,
          (unsigned)cfg.seed, ln_kind(mw, lay[k].first), 0.02);
      PD_CUDA(c, cudaGetLastError());
      c->launches += 1;
    }
    soff += c->wbytes[k];
  }
  if (src == nullptr) PD_CUDA(c, cudaStreamSynchronize(c->stream));
  pd::ModelW<W>* mwd = nullptr;
  PD_TRY(dalloc(c, &mwd, 1));
  PD_CUDA(c, cudaMemcpy(mwd, &mw, sizeof(mw), cudaMemcpyHostToDevice));
  c->mw_dev = mwd;

  pd::Bufs<W>& B = bufs<W>(c);
  const size_t R = D.rows, d = D.d;
  PD_TRY(dalloc(c, &B.ra, R * d)); PD_TRY(dalloc(c, &B.rb, R * d)); PD_TRY(dalloc(c, &B.rc, R * d));
  PD_TRY(dalloc(c, &B.xa, R * d)); PD_TRY(dalloc(c, &B.xb, R * d)); PD_TRY(dalloc(c, &B.xc, R * d));
  PD_TRY(dalloc(c, &B.q, R * d)); PD_TRY(dalloc(c, &B.k, R * d)); PD_TRY(dalloc(c, &B.v, R * d));
  PD_TRY(dalloc(c, &B.att, R * d));
  PD_TRY(dalloc(c, &B.ffh, R * (size_t)D.f));
  const size_t nb = (size_t)D.max_batch;
  PD_TRY(dalloc(c, &B.kself, (size_t)D.Ld * D.kv_pages * pd::kPageRows * d));
  PD_TRY(dalloc(c, &B.vself, (size_t)D.Ld * D.kv_pages * pd::kPageRows * d));
  PD_TRY(dalloc(c, &B.page_tab, nb * D.pt_ld));
  c->page_host.assign(nb * D.pt_ld, 0);
  PD_TRY(dalloc(c, &B.kcross, (size_t)D.Ld * nb * D.max_src * d));
  PD_TRY(dalloc(c, &B.vcross, (size_t)D.Ld * nb * D.max_src * d));
  PD_TRY(dalloc(c, &B.part, (size_t)c->grid * R));
  PD_TRY(dalloc(c, &B.st, 1));
  PD_TRY(dalloc(c, &B.trace, (size_t)D.max_tgt));
  PD_TRY(dalloc(c, &B.trace_tok, (size_t)D.max_tgt * D.max_tgt));
  PD_TRY(dalloc(c, &B.trace_prob, (size_t)D.max_tgt * D.max_tgt));
  PD_TRY(dalloc(c, &B.bar, 4));
  PD_TRY(dalloc(c, &B.src, nb * D.max_src));
  PD_TRY(dalloc(c, &B.dbg_tok, (size_t)D.max_tgt));
  PD_TRY(dalloc(c, &B.pos_tab, (size_t)D.max_keys * d));
  if (!cfg.learned_pos) {
    pd::sinusoid_kernel<<<c->n_sm, 256, 0, c->stream>>>(B.pos_tab, D.max_keys, (int)d);
    PD_CUDA(c, cudaGetLastError());
    PD_CUDA(c, cudaStreamSynchronize(c->stream));
    c->launches += 1;
  }
  PD_TRY(dalloc(c, &c->d_out_y, nb * D.max_tgt));
  PD_TRY(dalloc(c, &c->d_out_info, 4 * nb));
  PD_CUDA(c, cudaMemset(B.st, 0, sizeof(pd::DecState)));
  PD_CUDA(c, cudaMemset(B.bar, 0, 4 * sizeof(unsigned)));

  if constexpr (sizeof(W) == 2) {
    if (D.tc) PD_TRY(tc_resources(c, mw));
  }

  if (D.cl) PD_TRY(cl_resources<W>(c));
  c->smem = pd::smem_layout(D, sizeof(W)).total;
  if (D.cl) {                                 // the encoder runs the SIMT layout
    Dims De = D;
    De.cl = 0;
    c->smem = std::max(c->smem, pd::smem_layout(De, sizeof(W)).total);
  }
  if (D.tc && pd::smem_layout(D, sizeof(W)).ring_slots < 2)
    return fail(c, PD_EINVAL, "the tensor-core kernels' shared memory does not fit (max_tgt_len "
                              "or max_batch too large)");
  // the limit is per kernel function and shared by every context of the process: only raise it
  const void* fdec = kernel_fn<W>(false, D.tc != 0, D.cl != 0);
  const void* fenc = kernel_fn<W>(true, D.tc != 0);
  PD_TRY(raise_smem_limit(c, fdec));
  PD_TRY(raise_smem_limit(c, fenc));
  int nb1 = 0, nb2 = 0;
  PD_CUDA(c, cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb1, fdec, pd::kThreads, c->smem));
  PD_CUDA(c, cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb2, fenc, pd::kThreads, c->smem));
  if (nb1 < 1 || nb2 < 1) return fail(c, PD_EINVAL, "kernel does not fit on an SM (shared memory)");
  return PD_OK;
}

template <typename W>
pd::KParams<W> base_params(pd_ctx* c) {
  pd::KParams<W> P{};
  P.D = c->D;
  P.mw = static_cast<const pd::ModelW<W>*>(c->mw_dev);
  P.B = bufs<W>(c);
  for (int s = 0; s < pd::kMaxBatch; ++s) P.n_src_s[s] = c->n_src_slot[s];
  return P;
}

// reset_status: clear the status word first (every encode but the later ones of a batch, whose
// failures must survive until the batch is checked)
template <typename W>
pd_status launch(pd_ctx* c, bool encode, pd::KParams<W>& P, bool reset_status = true) {
  PD_CUDA(c, cudaMemsetAsync(bufs<W>(c).bar, 0, 4 * sizeof(unsigned), c->stream));
  if (encode && reset_status)
    PD_CUDA(c, cudaMemsetAsync(bufs<W>(c).st, 0, sizeof(pd::DecState), c->stream));
  if (c->D.tc) {                              // the kernel's tensor maps ride in its parameters
    const std::vector<CUtensorMap>& maps = encode ? c->enc_maps : c->dec_maps;
    std::memcpy(P.maps, maps.data(), maps.size() * sizeof(CUtensorMap));
  }
  void* args[] = {&P};
  const void* fn = kernel_fn<W>(encode, c->D.tc != 0, c->D.cl != 0);
  if (c->D.cl > 1 && !encode) {               // clusters of D.cl CTAs, cooperative (co-resident)
    cudaLaunchConfig_t lc{};
    lc.gridDim = dim3(c->cl_grid);
    lc.blockDim = dim3(pd::kThreads);
    lc.dynamicSmemBytes = c->smem;
    lc.stream = c->stream;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = (unsigned)c->D.cl;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeCooperative;
    at[1].val.cooperative = 1;
    lc.attrs = at;
    lc.numAttrs = 2;
    PD_CUDA(c, cudaLaunchKernelExC(&lc, fn, args));
    c->launches += 1;
    return PD_OK;
  }
  if (encode) P.D.cl = 0;                     // the cluster engine's encoder is the SIMT one
  // a kernel launched without clusters runs every CTA as a cluster of one (cluster_size 1)
  const int grid = (c->D.cl && !encode) ? c->cl_grid : c->grid;
  PD_CUDA(c, cudaLaunchCooperativeKernel(fn, dim3(grid), dim3(pd::kThreads), args, c->smem,
                                         c->stream));
  c->launches += 1;
  return PD_OK;
}

template <typename W>
pd_status encode_impl(pd_ctx* c, const int32_t* d_src, int n, int slot, bool reset_status) {
  pd::KParams<W> P = base_params<W>(c);
  P.n_src = n;
  P.enc_slot = slot;
  P.enc_tok = d_src;
  PD_TRY(launch<W>(c, true, P, reset_status));
  c->n_src_slot[slot] = n;
  return PD_OK;
}

pd_status assign_pages(pd_ctx* c, int n_sent, const int32_t* len, int len_all);

// max_len: per-sentence values (host), or nullptr for p->max_len everywhere
template <typename W>
pd_status decode_impl(pd_ctx* c, const pd_decode_params* p, int n_sent, const int32_t* max_len,
                      int32_t* d_y, int y_ld, int32_t* d_info) {
  pd::KParams<W> P = base_params<W>(c);
  P.init = pd::DecState{};
  P.init.method = p->method;
  P.init.b = p->b;
  P.init.h = p->h;
  P.init.stop_at_eos = p->stop_at_eos;
  P.init.max_passes = p->max_passes;
  P.init.stop_rule = p->stop_rule;
  P.init.init_rule = p->init;
  P.n_sent = n_sent;
  for (int s = 0; s < n_sent; ++s) P.max_len_s[s] = max_len ? max_len[s] : p->max_len;
  P.out_y = d_y;
  P.out_ld = y_ld;
  P.out_info = d_info;
  PD_TRY(assign_pages(c, n_sent, max_len, p->max_len));
  return launch<W>(c, false, P);
}

// A teacher-forced pass starts with a clear status word, so that a wait that gives up during
// it (PD_ETIMEOUT) is the only status the caller can read back afterwards (debug_status).
template <typename W>
pd_status debug_impl(pd_ctx* c, int len, float* d_logits) {
  PD_TRY(assign_pages(c, 1, nullptr, len));
  pd::KParams<W> P = base_params<W>(c);
  P.debug_len = len;
  P.logits = d_logits;
  PD_CUDA(c, cudaMemsetAsync(&bufs<W>(c).st->status, 0, sizeof(int), c->stream));
  return launch<W>(c, false, P);
}

// After the stream has been synchronised: the status a teacher-forced pass left (0 if it ran
// to the end).
pd_status debug_status(pd_ctx* c) {
  int st = 0;
  const pd::DecState* dst = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.st : c->bf.st;
  PD_CUDA(c, cudaMemcpy(&st, &dst->status, sizeof(int), cudaMemcpyDeviceToHost));
  if (st != 0) return fail(c, (pd_status)st, "the teacher-forced pass stopped early (a device "
                                             "wait gave up); no logits were returned");
  return PD_OK;
}

// Page tables of a decode: sentence s needs ceil(len_s / 16) pages of the self-attention
// key/value pool (positions 0..len_s - 1 are written); pages are handed out round robin over
// the sentences (page j of every sentence, then page j + 1, ...), so a sentence's pages are not
// contiguous in the pool.  The tables go to the device on the context stream.
pd_status assign_pages(pd_ctx* c, int n_sent, const int32_t* len, int len_all) {
  const Dims& D = c->D;
  long need = 0;
  int most = 0;
  for (int s = 0; s < n_sent; ++s) {
    const int l = len ? len[s] : len_all;
    const int np = (l + pd::kPageRows - 1) / pd::kPageRows;
    need += np;
    most = std::max(most, np);
  }
  if (need > D.kv_pages)
    return fail(c, PD_EINVAL, "the key/value page pool (kv_pages = " + std::to_string(D.kv_pages) +
                                  ") is smaller than the " + std::to_string(need) +
                                  " pages these sentences need");
  int next = 0;
  for (int j = 0; j < most; ++j)
    for (int s = 0; s < n_sent; ++s) {
      const int l = len ? len[s] : len_all;
      if (j < (l + pd::kPageRows - 1) / pd::kPageRows) c->page_host[(size_t)s * D.pt_ld + j] = next++;
    }
  int* dtab = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.page_tab : c->bf.page_tab;
  PD_CUDA(c, cudaMemcpyAsync(dtab, c->page_host.data(),
                             (size_t)n_sent * D.pt_ld * sizeof(int32_t), cudaMemcpyHostToDevice,
                             c->stream));
  return PD_OK;
}

// n_sent sentences (slots 0..n_sent-1), max_len per sentence (nullptr: p->max_len for all)
pd_status check_params(pd_ctx* c, const pd_decode_params* p, int n_sent = 1,
                       const int32_t* max_len = nullptr) {
  if (!p) return fail(c, PD_EINVAL, "params is NULL");
  if (p->method < PD_GREEDY || p->method > PD_HYBRID_GS_JACOBI) return fail(c, PD_EINVAL, "method");
  if ((p->method == PD_GS_JACOBI || p->method == PD_HYBRID_GS_JACOBI) && p->b < 1)
    return fail(c, PD_EINVAL, "b must be >= 1");
  if (p->max_passes < 0) return fail(c, PD_EINVAL, "max_passes must be >= 0");
  if (p->stop_rule != PD_STOP_UNCHANGED && p->stop_rule != PD_STOP_PREFIX &&
      p->stop_rule != PD_STOP_SUFFIX)
    return fail(c, PD_EINVAL, "stop_rule");
  if (p->init != PD_INIT_PAD && p->init != PD_INIT_LAST) return fail(c, PD_EINVAL, "init");
  if (n_sent < 1 || n_sent > c->D.max_batch) return fail(c, PD_EINVAL, "n_sent must be in [1, max_batch]");
  long rows = 0;                                  // rows of the widest pass
  for (int s = 0; s < n_sent; ++s) {
    const int m = max_len ? max_len[s] : p->max_len;
    if (m < 1 || m > c->cfg.max_tgt_len)
      return fail(c, PD_EINVAL, "max_len must be in [1, max_tgt_len]");
    if (c->cfg.learned_pos && m > c->cfg.max_pos)
      return fail(c, PD_EINVAL, "max_len exceeds the learned position table");
    const int b_eff = p->method == PD_GREEDY ? 1 : (p->method == PD_JACOBI ? m : p->b);
    rows += b_eff < m ? b_eff : m;
  }
  if (rows > c->D.rows) return fail(c, PD_EINVAL, "the sentences' blocks exceed the rows of a pass");
  if (c->n_encoded < n_sent) return fail(c, PD_ESTATE, "pd_decode before pd_encode");
  return PD_OK;
}

}  // namespace

// ============================================================================================
// C ABI
// ============================================================================================

static pd_status static_logits_lookup(pd_ctx* c);

// Reason of this thread's last failed pd_create (read through pd_last_error(NULL)).
static thread_local std::string g_create_err;

extern "C" {

size_t pd_weights_nbytes(const pd_config* cfg) {
  if (!valid_config(cfg, nullptr)) return 0;
  return blob_elems(*cfg) * wsize(*cfg);
}

pd_status pd_create(const pd_config* cfg, const void* weights, size_t nbytes, void* stream,
                    pd_ctx** out) {
  g_create_err.clear();
  if (!out) { g_create_err = "out is NULL"; return PD_EINVAL; }
  *out = nullptr;
  std::string why;
  if (!valid_config(cfg, &why)) { g_create_err = "invalid config: " + why; return PD_EINVAL; }
  if (!weights && nbytes != 0) {
    g_create_err = "weights is NULL: nbytes must be 0 (the library draws the weights)";
    return PD_EINVAL;
  }
  if (weights && nbytes != pd_weights_nbytes(cfg)) {
    g_create_err = "nbytes is " + std::to_string(nbytes) + ", the blob of this config has " +
                   std::to_string(pd_weights_nbytes(cfg));
    return PD_EINVAL;
  }
  pd_ctx* c = new pd_ctx();
  c->cfg = *cfg;
  Dims& D = c->D;
  D.d = cfg->d_model; D.H = cfg->n_heads; D.dh = cfg->d_model / cfg->n_heads; D.f = cfg->d_ff;
  D.Le = cfg->n_enc_layers; D.Ld = cfg->n_dec_layers; D.V = cfg->vocab;
  D.act = cfg->activation; D.pre_ln = cfg->pre_ln ? 1 : 0; D.learned_pos = cfg->learned_pos ? 1 : 0;
  D.max_pos = cfg->learned_pos ? cfg->max_pos : 1;
  D.pad = cfg->pad_id; D.eos = cfg->eos_id; D.bos = cfg->bos_id;
  D.eps = cfg->ln_eps; D.emb_scale = sqrtf((float)cfg->d_model);
  D.max_src = cfg->max_src_len; D.max_tgt = cfg->max_tgt_len;
  D.max_keys = D.max_src > D.max_tgt ? D.max_src : D.max_tgt;
  D.max_batch = cfg->max_batch > 1 ? cfg->max_batch : 1;
  D.pt_ld = (D.max_tgt + pd::kPageRows - 1) / pd::kPageRows;
  D.kv_pages = cfg->kv_pages > 0 ? cfg->kv_pages : D.max_batch * D.pt_ld;
  const long batch_rows = std::min<long>((long)D.max_batch * D.max_tgt, pd::kMaxPassRows);
  D.rows = (int)std::max<long>(D.max_keys, batch_rows);
  D.tc = cfg->dtype == PD_DTYPE_BF16 && cfg->gemm_engine == PD_ENGINE_TENSOR;
  D.cl = cfg->gemm_engine == PD_ENGINE_CLUSTER ? (cfg->cluster_size > 0 ? cfg->cluster_size : 8) : 0;
  c->blob_bytes = pd_weights_nbytes(cfg);
  pd_status s = PD_OK;
  cudaError_t e = cudaGetDevice(&c->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&c->n_sm, cudaDevAttrMultiProcessorCount, c->device);
  int coop = 0;
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, c->device);
  if (e != cudaSuccess || !coop) {
    g_create_err = e != cudaSuccess ? std::string("device query: ") + cudaGetErrorString(e)
                                    : "the device has no cooperative launch";
    pd_destroy(c);
    return PD_ECUDA;
  }
  c->grid = c->n_sm;
  if (stream) {
    c->stream = static_cast<cudaStream_t>(stream);
  } else {
    if (cudaStreamCreateWithFlags(&c->stream, cudaStreamNonBlocking) != cudaSuccess) {
      g_create_err = "cudaStreamCreateWithFlags failed";
      pd_destroy(c);
      return PD_ECUDA;
    }
    c->own_stream = true;
  }
  s = cfg->dtype == PD_DTYPE_BF16 ? create_impl<__nv_bfloat16>(c, weights)
                                  : create_impl<float>(c, weights);
  if (s == PD_OK) s = static_logits_lookup(c);
  if (s != PD_OK) {
    g_create_err = c->err;
    pd_destroy(c);
    return s;
  }
  *out = c;
  return PD_OK;
}

pd_status pd_export_weights(pd_ctx* c, void* dst, size_t nbytes) {
  if (!c) return PD_EINVAL;
  if (!dst || nbytes != c->blob_bytes) return fail(c, PD_EINVAL, "dst size must equal the blob size");
  unsigned char* o = static_cast<unsigned char*>(dst);
  size_t off = 0;
  for (size_t k = 0; k < c->woff.size(); ++k) {
    PD_CUDA(c, cudaMemcpy(o + off, static_cast<unsigned char*>(c->wdev) + c->woff[k], c->wbytes[k],
                          cudaMemcpyDeviceToHost));
    off += c->wbytes[k];
  }
  return PD_OK;
}

pd_status pd_encode_device(pd_ctx* c, const int32_t* d_src, int n_src) {
  if (!c) return PD_EINVAL;
  if (!d_src || n_src < 1 || n_src > c->cfg.max_src_len)
    return fail(c, PD_EINVAL, "n_src must be in [1, max_src_len]");
  if (c->cfg.learned_pos && n_src > c->cfg.max_pos)
    return fail(c, PD_EINVAL, "n_src exceeds the learned position table");
  c->n_encoded = 0;
  PD_TRY(c->cfg.dtype == PD_DTYPE_BF16 ? encode_impl<__nv_bfloat16>(c, d_src, n_src, 0, true)
                                       : encode_impl<float>(c, d_src, n_src, 0, true));
  c->n_encoded = 1;
  return PD_OK;
}

pd_status pd_encode(pd_ctx* c, const int32_t* src, int n_src) {
  if (!c) return PD_EINVAL;
  if (!src || n_src < 1 || n_src > c->cfg.max_src_len)
    return fail(c, PD_EINVAL, "n_src must be in [1, max_src_len]");
  for (int k = 0; k < n_src; ++k)
    if (src[k] < 0 || src[k] >= c->cfg.vocab) return fail(c, PD_EINVAL, "source id out of range");
  int32_t* dsrc = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.src : c->bf.src;
  PD_CUDA(c, cudaMemcpyAsync(dsrc, src, n_src * sizeof(int32_t), cudaMemcpyHostToDevice, c->stream));
  PD_TRY(pd_encode_device(c, dsrc, n_src));
  PD_CUDA(c, cudaStreamSynchronize(c->stream));
  int st = 0;
  pd::DecState* dst = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.st : c->bf.st;
  PD_CUDA(c, cudaMemcpy(&st, &dst->status, sizeof(int), cudaMemcpyDeviceToHost));
  if (st != 0) {
    c->n_encoded = 0;
    return fail(c, (pd_status)st, "encoder kernel reported a failure");
  }
  return PD_OK;
}

pd_status pd_encode_batch_device(pd_ctx* c, const int32_t* d_src, const int32_t* offsets,
                                 int n_sent) {
  if (!c) return PD_EINVAL;
  if (!d_src || !offsets || n_sent < 1 || n_sent > c->D.max_batch)
    return fail(c, PD_EINVAL, "d_src, offsets and n_sent in [1, max_batch] are required");
  for (int s = 0; s < n_sent; ++s) {
    const int n = offsets[s + 1] - offsets[s];
    if (offsets[s] < 0 || n < 1 || n > c->cfg.max_src_len)
      return fail(c, PD_EINVAL, "every sentence length must be in [1, max_src_len]");
    if (c->cfg.learned_pos && n > c->cfg.max_pos)
      return fail(c, PD_EINVAL, "a sentence exceeds the learned position table");
  }
  c->n_encoded = 0;
  for (int s = 0; s < n_sent; ++s) {
    const int n = offsets[s + 1] - offsets[s];
    PD_TRY(c->cfg.dtype == PD_DTYPE_BF16
               ? encode_impl<__nv_bfloat16>(c, d_src + offsets[s], n, s, s == 0)
               : encode_impl<float>(c, d_src + offsets[s], n, s, s == 0));
  }
  c->n_encoded = n_sent;
  return PD_OK;
}

pd_status pd_encode_batch(pd_ctx* c, const int32_t* src, const int32_t* offsets, int n_sent) {
  if (!c) return PD_EINVAL;
  if (!src || !offsets || n_sent < 1 || n_sent > c->D.max_batch)
    return fail(c, PD_EINVAL, "src, offsets and n_sent in [1, max_batch] are required");
  if (offsets[0] != 0) return fail(c, PD_EINVAL, "offsets[0] must be 0");
  for (int s = 0; s < n_sent; ++s) {
    const int n = offsets[s + 1] - offsets[s];
    if (n < 1 || n > c->cfg.max_src_len)
      return fail(c, PD_EINVAL, "every sentence length must be in [1, max_src_len]");
  }
  const int total = offsets[n_sent];
  for (int k = 0; k < total; ++k)
    if (src[k] < 0 || src[k] >= c->cfg.vocab) return fail(c, PD_EINVAL, "source id out of range");
  int32_t* dsrc = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.src : c->bf.src;
  PD_CUDA(c, cudaMemcpyAsync(dsrc, src, total * sizeof(int32_t), cudaMemcpyHostToDevice, c->stream));
  PD_TRY(pd_encode_batch_device(c, dsrc, offsets, n_sent));
  PD_CUDA(c, cudaStreamSynchronize(c->stream));
  int st = 0;
  pd::DecState* dst = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.st : c->bf.st;
  PD_CUDA(c, cudaMemcpy(&st, &dst->status, sizeof(int), cudaMemcpyDeviceToHost));
  if (st != 0) {
    c->n_encoded = 0;
    return fail(c, (pd_status)st, "encoder kernel reported a failure");
  }
  return PD_OK;
}

pd_status pd_decode_device(pd_ctx* c, const pd_decode_params* p, int32_t* d_y, int32_t* d_info) {
  if (!c) return PD_EINVAL;
  PD_TRY(check_params(c, p));
  if (!d_y || !d_info) return fail(c, PD_EINVAL, "d_y and d_info are required");
  return c->cfg.dtype == PD_DTYPE_BF16
             ? decode_impl<__nv_bfloat16>(c, p, 1, nullptr, d_y, p->max_len, d_info)
             : decode_impl<float>(c, p, 1, nullptr, d_y, p->max_len, d_info);
}

pd_status pd_decode_batch_device(pd_ctx* c, const pd_decode_params* p, int n_sent,
                                 const int32_t* max_len, int32_t* d_y, int y_ld, int32_t* d_info) {
  if (!c) return PD_EINVAL;
  PD_TRY(check_params(c, p, n_sent, max_len));
  if (!d_y || !d_info) return fail(c, PD_EINVAL, "d_y and d_info are required");
  for (int s = 0; s < n_sent; ++s)
    if ((max_len ? max_len[s] : p->max_len) > y_ld) return fail(c, PD_EINVAL, "y_ld < max_len");
  return c->cfg.dtype == PD_DTYPE_BF16
             ? decode_impl<__nv_bfloat16>(c, p, n_sent, max_len, d_y, y_ld, d_info)
             : decode_impl<float>(c, p, n_sent, max_len, d_y, y_ld, d_info);
}

pd_status pd_decode_batch(pd_ctx* c, const pd_decode_params* p, int n_sent,
                          const int32_t* max_len, int32_t* y, int y_ld, int32_t* n_y,
                          int32_t* n_iters) {
  if (!c) return PD_EINVAL;
  if (!y || !n_y || !n_iters) return fail(c, PD_EINVAL, "y, n_y and n_iters are required");
  const int ld = c->cfg.max_tgt_len;
  PD_TRY(pd_decode_batch_device(c, p, n_sent, max_len, c->d_out_y, ld, c->d_out_info));
  std::vector<int32_t> info(4 * (size_t)n_sent);
  PD_CUDA(c, cudaMemcpyAsync(info.data(), c->d_out_info, info.size() * sizeof(int32_t),
                             cudaMemcpyDeviceToHost, c->stream));
  PD_CUDA(c, cudaStreamSynchronize(c->stream));
  const int w = std::min(y_ld, ld);
  PD_CUDA(c, cudaMemcpy2D(y, y_ld * sizeof(int32_t), c->d_out_y, ld * sizeof(int32_t),
                          w * sizeof(int32_t), n_sent, cudaMemcpyDeviceToHost));
  int first_bad = 0;
  for (int s = 0; s < n_sent; ++s) {
    const int m = max_len ? max_len[s] : p->max_len;
    n_y[s] = info[4 * s] < 0 ? 0 : std::min(info[4 * s], m);
    n_iters[s] = info[4 * s + 1];
    if (!first_bad && info[4 * s + 2] != 0) first_bad = info[4 * s + 2];
  }
  if (first_bad != 0)
    return fail(c, (pd_status)first_bad, first_bad == PD_ENOTCONV ? "pass budget exhausted"
                                         : first_bad == PD_ENAN ? "NaN in the logits"
                                         : "decode kernel reported a failure");
  return PD_OK;
}

pd_status pd_decode(pd_ctx* c, const pd_decode_params* p, int32_t* y, int* n_y, int* n_iters,
                    pd_trace_step* trace, int32_t* trace_tokens, float* trace_probs, int trace_cap,
                    int* n_trace) {
  if (!c) return PD_EINVAL;
  PD_TRY(check_params(c, p));
  if (!y || !n_y || !n_iters) return fail(c, PD_EINVAL, "y, n_y and n_iters are required");
  if (trace && (trace_cap < 0 || !n_trace)) return fail(c, PD_EINVAL, "trace needs trace_cap and n_trace");
  PD_TRY(pd_decode_device(c, p, c->d_out_y, c->d_out_info));
  int32_t info[4];
  PD_CUDA(c, cudaMemcpyAsync(info, c->d_out_info, sizeof(info), cudaMemcpyDeviceToHost, c->stream));
  PD_CUDA(c, cudaStreamSynchronize(c->stream));
  const int ny = info[0] < 0 ? 0 : (info[0] > p->max_len ? p->max_len : info[0]);
  if (ny > 0)
    PD_CUDA(c, cudaMemcpy(y, c->d_out_y, ny * sizeof(int32_t), cudaMemcpyDeviceToHost));
  *n_y = ny;
  *n_iters = info[1];
  if (trace) {
    const int D_tgt = c->cfg.max_tgt_len;
    const int nt = info[3] < trace_cap ? info[3] : trace_cap;
    pd_trace_step* dtr = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.trace : c->bf.trace;
    int* dtt = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.trace_tok : c->bf.trace_tok;
    float* dtp = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.trace_prob : c->bf.trace_prob;
    if (nt > 0) {
      PD_CUDA(c, cudaMemcpy(trace, dtr, nt * sizeof(pd_trace_step), cudaMemcpyDeviceToHost));
      if (trace_tokens || trace_probs) {
        // device rows have stride max_tgt_len; the caller's rows have stride max_len
        PD_CUDA(c, cudaMemcpy2D(trace_tokens ? (void*)trace_tokens : (void*)trace_probs,
                                p->max_len * sizeof(int32_t), trace_tokens ? (void*)dtt : (void*)dtp,
                                D_tgt * sizeof(int32_t), p->max_len * sizeof(int32_t), nt,
                                cudaMemcpyDeviceToHost));
        if (trace_tokens && trace_probs)
          PD_CUDA(c, cudaMemcpy2D(trace_probs, p->max_len * sizeof(float), dtp, D_tgt * sizeof(float),
                                  p->max_len * sizeof(float), nt, cudaMemcpyDeviceToHost));
      }
    }
    *n_trace = nt;
  }
  const int st = info[2];
  if (st != 0) return fail(c, (pd_status)st, st == PD_ENOTCONV ? "pass budget exhausted"
                                               : st == PD_ENAN ? "NaN in the logits"
                                               : "decode kernel reported a failure");
  return PD_OK;
}

pd_status pd_debug_logits(pd_ctx* c, const int32_t* y_in, int len, float* logits) {
  if (!c) return PD_EINVAL;
  if (!y_in || !logits || len < 1 || len > c->cfg.max_tgt_len)
    return fail(c, PD_EINVAL, "len must be in [1, max_tgt_len]");
  if (c->cfg.learned_pos && len > c->cfg.max_pos) return fail(c, PD_EINVAL, "len exceeds max_pos");
  for (int k = 0; k < len; ++k)
    if (y_in[k] < 0 || y_in[k] >= c->cfg.vocab) return fail(c, PD_EINVAL, "token id out of range");
  if (c->n_encoded < 1) return fail(c, PD_ESTATE, "pd_debug_logits before pd_encode");
  int* dtok = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.dbg_tok : c->bf.dbg_tok;
  PD_CUDA(c, cudaMemcpyAsync(dtok, y_in, len * sizeof(int32_t), cudaMemcpyHostToDevice, c->stream));
  float* dl = nullptr;
  const size_t nb = (size_t)len * c->cfg.vocab * sizeof(float);
  PD_CUDA(c, cudaMalloc(&dl, nb));
  pd_status s = c->cfg.dtype == PD_DTYPE_BF16 ? debug_impl<__nv_bfloat16>(c, len, dl)
                                               : debug_impl<float>(c, len, dl);
  cudaError_t e = s == PD_OK ? cudaStreamSynchronize(c->stream) : cudaSuccess;
  if (s == PD_OK && e == cudaSuccess) s = debug_status(c);
  if (s == PD_OK && e == cudaSuccess) e = cudaMemcpy(logits, dl, nb, cudaMemcpyDeviceToHost);
  cudaFree(dl);
  if (s != PD_OK) return s;
  if (e != cudaSuccess) return fail(c, PD_ECUDA, std::string("debug logits: ") + cudaGetErrorString(e));
  return PD_OK;
}

}  // extern "C"

// ------------------------------------------------------------------------------------------
// pd_debug_logits_static: the teacher-forced logits without any device allocation
// ------------------------------------------------------------------------------------------
//
// pd_debug_logits stages the logits in a device buffer it allocates for each call.  Callers
// that may not allocate device memory (a process whose memory is pooled by another owner, a
// code path running under an allocator lock, or a program that must not grow its footprint
// after start-up) use this variant: the staging buffer is a fixed array in the library's own
// device image, loaded once per GPU with the module and kept until the process exits.

namespace {

constexpr size_t kStaticLogitsFloats = (size_t)1 << 20;   // 4 MiB: len * vocab <= 1,048,576

}  // namespace

// In host code this name stands for the array; its device address comes from
// cudaGetSymbolAddress, looked up by static_logits_lookup when a context is created.
static __device__ __align__(256) float g_static_logits[kStaticLogitsFloats];

// Device address of g_static_logits on the context's device (current while pd_create runs),
// kept in the context: a context never outlives its device's primary context, so the address
// stays valid for every later call on it.
static pd_status static_logits_lookup(pd_ctx* c) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_static_logits);
  if (e != cudaSuccess || p == nullptr)
    return fail(c, PD_ECUDA, std::string("cudaGetSymbolAddress(g_static_logits): ") +
                                 cudaGetErrorString(e));
  c->static_logits = static_cast<float*>(p);
  return PD_OK;
}

extern "C" {

pd_status pd_debug_logits_static(pd_ctx* c, const int32_t* y_in, int len, float* logits) {
  if (!c) return PD_EINVAL;
  if (!y_in || !logits || len < 1 || len > c->cfg.max_tgt_len)
    return fail(c, PD_EINVAL, "len must be in [1, max_tgt_len]");
  if ((size_t)len * (size_t)c->cfg.vocab > kStaticLogitsFloats)
    return fail(c, PD_EINVAL, "len * vocab exceeds the static logits buffer (1,048,576 floats)");
  if (c->cfg.learned_pos && len > c->cfg.max_pos) return fail(c, PD_EINVAL, "len exceeds max_pos");
  for (int k = 0; k < len; ++k)
    if (y_in[k] < 0 || y_in[k] >= c->cfg.vocab) return fail(c, PD_EINVAL, "token id out of range");
  if (c->n_encoded < 1) return fail(c, PD_ESTATE, "pd_debug_logits_static before pd_encode");
  float* dl = c->static_logits;
  int* dtok = c->cfg.dtype == PD_DTYPE_BF16 ? c->bb.dbg_tok : c->bf.dbg_tok;
  PD_CUDA(c, cudaMemcpyAsync(dtok, y_in, len * sizeof(int32_t), cudaMemcpyHostToDevice, c->stream));
  // every element of the [len][vocab] region is written by the kernel: nothing to clear
  PD_TRY(c->cfg.dtype == PD_DTYPE_BF16 ? debug_impl<__nv_bfloat16>(c, len, dl)
                                       : debug_impl<float>(c, len, dl));
  PD_CUDA(c, cudaStreamSynchronize(c->stream));
  PD_TRY(debug_status(c));
  PD_CUDA(c, cudaMemcpyAsync(logits, dl, (size_t)len * c->cfg.vocab * sizeof(float),
                             cudaMemcpyDeviceToHost, c->stream));
  PD_CUDA(c, cudaStreamSynchronize(c->stream));
  return PD_OK;
}

pd_status pd_debug_wait_timeout(pd_ctx* c, uint64_t limit_ns, int* status) {
  if (!c) return PD_EINVAL;
  if (!status || limit_ns == 0 || limit_ns > 10000000000ull)
    return fail(c, PD_EINVAL, "limit_ns must be in (0, 1e10] and status non-NULL");
  unsigned* words = nullptr;   // [0] counter, [1] abort flag, [2] unused, [3] the status
  PD_CUDA(c, cudaMalloc(&words, 4 * sizeof(unsigned)));
  pd_status st = PD_OK;
  int host[4] = {0, 0, 0, 0};
  if (cudaMemsetAsync(words, 0, 4 * sizeof(unsigned), c->stream) != cudaSuccess) st = PD_ECUDA;
  if (st == PD_OK) {
    pd::wait_probe_kernel<<<1, 32, 0, c->stream>>>(words, reinterpret_cast<int*>(words + 3),
                                                   (unsigned long long)limit_ns);
    c->launches += 1;
    if (cudaGetLastError() != cudaSuccess ||
        cudaMemcpyAsync(host, words, sizeof(host), cudaMemcpyDeviceToHost, c->stream) !=
            cudaSuccess ||
        cudaStreamSynchronize(c->stream) != cudaSuccess)
      st = PD_ECUDA;
  }
  cudaFree(words);
  if (st != PD_OK) return fail(c, st, "wait probe failed");
  *status = host[3];
  return host[1] != 0u ? PD_OK : fail(c, PD_ESTATE, "the probe's abort flag was not raised");
}

void* pd_stream(pd_ctx* c) { return c ? (void*)c->stream : nullptr; }


int64_t pd_launch_count(const pd_ctx* c) { return c ? c->launches : 0; }

const char* pd_last_error(const pd_ctx* c) { return c ? c->err.c_str() : g_create_err.c_str(); }

void pd_destroy(pd_ctx* c) {
  if (!c) return;
  if (c->stream) cudaStreamSynchronize(c->stream);
  for (void* p : c->allocs) cudaFree(p);
  if (c->own_stream && c->stream) cudaStreamDestroy(c->stream);
  delete c;
}

}  // extern "C"

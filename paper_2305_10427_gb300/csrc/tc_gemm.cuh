// Tensor-core (tcgen05 / TMEM / TMA) GEMM phase of the bf16 decoder and encoder.
//
// A GEMM phase computes Y[M][N] = epilogue(X[M][K] . W[N][K]^T + bias) for the M rows of a
// pass.  The products run on the 5th-generation tensor cores with the operands swapped: a tile
// of 128 weight rows (output features) is the MMA's A operand, brought into shared memory by
// TMA (cp.async.bulk.tensor, 128-byte swizzle, boxes of 128 rows x 64 K), and the pass's token
// rows are the B operand, 16 rows per MMA (kind::f16, M = 128, N = 16, K = 16), staged into
// shared memory by the CTA's threads (LayerNorm / embedding prologue fused).  Accumulators live
// in tensor memory and are read back with tcgen05.ld for the fused epilogue.
//
// Batch invariance.  Every MMA has the same shape (N = 16 token rows) and every output
// element accumulates its K products in the same order (K-blocks of 64 ascending, K = 16 steps
// inside); a K split across CTAs (K > 512) is summed in ascending split order; so the value of
// a row's output does not depend on how many rows the pass carries or where the row sits, and
// every decoding method returns exactly the greedy tokens.
//
// Work division.  A phase has tiles = ceil(N / 128) output tiles, each split into S = K / 512
// K-slices (S = 1 for K <= 512 and for the LM head, whose argmax needs whole dot products):
// items = tiles x S, item i of phase g going to CTA (i + off_g) mod grid, where off_g counts the
// items of the pass's earlier GEMM phases, so consecutive phases land on different CTAs.  A
// CTA's sequence of weight K-blocks over a pass depends on N and K only, so one thread streams
// them through a ring of shared-memory slots ahead of use (while the CTA waits at grid
// barriers); an item's MMAs then find their weights resident.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "pd_device.cuh"

namespace pd {

constexpr int kRingMax = 8;            // weight slots (16 KB each)
constexpr int kTileN = 128;            // output features per tile (the MMA's M)
constexpr int kKBlock = 64;            // K elements of one TMA box (128 bytes of bf16)
constexpr int kSlotBytes = kTileN * kKBlock * 2;
constexpr int kRowTile = 16;           // token rows per MMA (the MMA's N)
constexpr int kBBytes = 64 * 1024;     // staged token rows (B operand)
constexpr int kKSliceMax = 512;        // K per item of a split phase
constexpr int kMaxChunk = 128;         // token rows per chunk (B buffer, MMA N, TMEM columns)
constexpr int kEpiLd = kTileN + 4;     // floats per row of the epilogue tile
constexpr int kEpiBytes = kRowTile * kEpiLd * 4;
constexpr int kAccs = 4;               // independent accumulators per item (K-block kb -> kb % 4)
constexpr int kTmemCols = kAccs * kMaxChunk;
constexpr int kMaxGemmPhases = 8 * kMaxLayers + 1;
constexpr int kCounterSlots = 8192;    // split-K arrival counters (tile x chunk)

// Kinds of phase sequences the weight stream walks.
enum TcKind : int { TC_DECODE = 0, TC_ENCODE = 1 };

// Decoder GEMM phase types, in pass order (phase g = 6 l + type, then the LM head at 6 Ld).
enum : int { TD_QKV = 0, TD_O = 1, TD_QC = 2, TD_OC = 3, TD_FFN1 = 4, TD_FFN2 = 5 };
// Encoder GEMM phase types (phase g = 4 l + type for l < Le, then g = 4 Le + l: the cross K/V
// projection of decoder layer l).
enum : int { TE_QKV = 0, TE_O = 1, TE_FFN1 = 2, TE_FFN2 = 3 };

// Each kernel receives, among its parameters, one TMA tensor map per GEMM phase of its phase
// sequence (index = the phase's GEMM index g): parameter space is read through the constant
// cache, so issuing a TMA load does not wait for a descriptor fetch from device memory.
constexpr int kMaxKernelMaps = 6 * kMaxLayers + 1;

struct Geom {
  int tmap;          // index of the phase's tensor map among the kernel's parameters
  int N, K, S, KS;   // outputs, inputs, K split, K per item
  int RC;            // token rows per chunk
  int tiles, items;
};

// One GEMM phase as this CTA sees it (computed once per kernel, in shared memory): N outputs,
// items = tiles x S, S K-slices of kbs K-blocks, first = this CTA's first unit, at most rtmax
// 16-row tiles per chunk of token rows (the staged B operand's capacity).  A pass of M rows
// cuts the rows into chunks (cl_chunks below); its units are (chunk, item) pairs, unit u being
// item u mod items of chunk u / items, and this CTA takes units first, first + grid, ...
struct PInfo {
  int N, items;
  short first, nj0;              // nj0: this CTA's units of chunk 0 (u < items)
  unsigned char S, kbs, rtmax, pad;
};

// Row chunks of a pass of M rows for phase `in`: enough chunks that the units (items x chunks)
// spread over the grid, at most M / 16 of them (16-row tiles), and none larger than rtmax
// tiles; rc = rows per chunk (a multiple of 16), nch = chunks, nj = this CTA's units.  A row's
// arithmetic does not depend on the chunking (every MMA covers 16-row tiles with the same K
// order), so the choice may follow M.  M = 0 (rows not known yet): chunk 0 only.
__device__ __forceinline__ void tc_chunks(const PInfo& in, int M, int grid, int& rc, int& nch,
                                          int& nj) {
  if (M <= 0) {
    rc = kRowTile; nch = 1; nj = in.nj0;
    return;
  }
  const int rt = (M + kRowTile - 1) / kRowTile;             // 16-row tiles of the pass
  int c = (grid + in.items - 1) / in.items;                  // chunks that fill the grid
  const int cmin = (rt + in.rtmax - 1) / in.rtmax;
  c = c < cmin ? cmin : (c > rt ? rt : c);
  const int rtc = (rt + c - 1) / c;
  rc = rtc * kRowTile;
  nch = (M + rc - 1) / rc;
  const int units = in.items * nch;
  nj = in.first < units ? (units - in.first + grid - 1) / grid : 0;
}

// Per-CTA state of the tensor-core path (shared memory).  Only thread 0 touches the stream
// cursor; every thread reads acc_n.
struct TcState {
  unsigned long long full[kRingMax];   // slot filled (TMA transaction bytes)
  unsigned long long empty[kRingMax];  // slot read by its MMAs (tcgen05.commit)
  unsigned long long acc;              // an item's MMAs are done (tcgen05.commit)
  uint32_t tmem;                       // tensor-memory base address
  int ring, ring_sh;                   // slots in use (a power of two) and its log2
  int kind, n_g;                       // phase sequence and its GEMM phase count
  PInfo info[kMaxGemmPhases];          // the kernel's GEMM phases as this CTA sees them
  // weight stream cursor: phase, unit of this CTA, K-block; sequence number; rows of the pass
  // it walks; keep streaming into the next pass; blocks past the current pass are speculative
  int p_g, p_j, p_kb, p_seq, p_M, p_open, p_spec;
  int c_seq;                           // K-blocks consumed
  // this pass's plan (tc_plan): this CTA's units and row tiles per chunk of every GEMM phase
  short pj[kMaxGemmPhases];
  unsigned char prt[kMaxGemmPhases];
  int acc_n;                           // items whose accumulator has been read
  int last;                            // split-K: this CTA sums the tile's partials
  int err;                             // a bounded wait gave up
};

template <typename W>
__device__ __forceinline__ TcState& smem_tc() {
  __shared__ TcState s;
  return s;
}

// ------------------------------------------------------------------------------------------
// PTX wrappers
// ------------------------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(unsigned long long* b, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(b)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(unsigned long long* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(b)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(unsigned long long* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(b)) : "memory");
}

// Non-blocking test of the phase with the given parity.
__device__ __forceinline__ bool mbar_test(unsigned long long* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(b)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait for a phase; false (and the CTA's error flag) if it did not complete in time.
__device__ __forceinline__ bool mbar_wait(unsigned long long* b, uint32_t parity, int* err,
                                          unsigned long long limit_ns = kWaitNs) {
  if (mbar_test(b, parity)) return true;
  const unsigned long long t0 = globaltimer_ns();
  for (unsigned n = 1;; ++n) {
    if (mbar_test(b, parity)) return true;
    if ((n & 63u) == 0u && globaltimer_ns() - t0 > limit_ns) {
      *err = 1;
      return false;
    }
  }
}

// 2-D tile load of a weight box (x = K element offset, y = row offset) into shared memory,
// completing `bytes` transaction bytes on mbarrier b.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map,
                                            unsigned long long* b, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(b)), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Whole warp.
__device__ __forceinline__ void tmem_alloc(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// D[tmem] (+)= A[smem desc] . B[smem desc]^T, bf16 inputs, fp32 accumulation.
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on mbarrier b when every tcgen05 operation this thread issued so far is done.
__device__ __forceinline__ void mma_commit(unsigned long long* b) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::
                   "r"(smem_u32(b))
               : "memory");
}

// This warp's 32 lanes (lane base 32 (warp % 4)), 16 consecutive 32-bit columns from col.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor of a K-major operand in the 128-byte swizzle layout: rows of
// 128 bytes (64 bf16 of K), 8-row atoms of 1024 bytes stacked along M / N (stride 1024).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);          // start address
  d |= (uint64_t)1 << 16;                           // leading byte offset (unused here)
  d |= (uint64_t)(1024 >> 4) << 32;                 // stride byte offset
  d |= (uint64_t)1 << 46;                           // descriptor version
  d |= (uint64_t)2 << 61;                           // 128-byte swizzle
  return d;
}

// Instruction descriptor: kind::f16 with bf16 A and B, fp32 D, both K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

// Byte offset of token row r, K element kk (within the item's K-slice) in the staged B
// operand: [K-block][16-row tile][16 rows x 128 bytes], 16-byte chunks XOR-swizzled by r % 8.
__device__ __forceinline__ uint32_t b_offset(int r, int kk, int rtiles) {
  const int kb = kk >> 6, c = (kk & 63) >> 3;
  return (uint32_t)(kb * rtiles * 2048 + (r >> 4) * 2048 + (r & 15) * 128 +
                    ((c ^ (r & 7)) << 4) + (kk & 7) * 2);
}

// ------------------------------------------------------------------------------------------
// geometry of the GEMM phases
// ------------------------------------------------------------------------------------------

__host__ __device__ inline Geom make_geom(int tmap, int N, int K, bool lm_head) {
  Geom g;
  g.tmap = tmap;
  g.N = N;
  g.K = K;
  // K is a multiple of 256: slices of 512 where they divide K, else of 256
  g.S = (lm_head || K <= kKSliceMax) ? 1 : (K % kKSliceMax == 0 ? K / kKSliceMax : K / 256);
  g.KS = K / g.S;
  int rc = kBBytes / (2 * g.KS);
  rc = rc / kRowTile * kRowTile;
  g.RC = rc > kMaxChunk ? kMaxChunk : rc;
  g.tiles = (N + kTileN - 1) / kTileN;
  g.items = g.tiles * g.S;
  return g;
}

__host__ __device__ inline int gemm_phase_count(const Dims& D, int kind) {
  return kind == TC_DECODE ? 6 * D.Ld + 1 : 4 * D.Le + D.Ld;
}

__host__ __device__ inline Geom gemm_geom(const Dims& D, int kind, int g) {
  const int d = D.d, f = D.f;
  if (kind == TC_DECODE) {
    if (g == 6 * D.Ld) return make_geom(g, D.V, d, true);
    switch (g % 6) {
      case TD_QKV: return make_geom(g, 3 * d, d, false);
      case TD_O: return make_geom(g, d, d, false);
      case TD_QC: return make_geom(g, d, d, false);
      case TD_OC: return make_geom(g, d, d, false);
      case TD_FFN1: return make_geom(g, f, d, false);
      default: return make_geom(g, d, f, false);
    }
  }
  if (g >= 4 * D.Le) return make_geom(g, 2 * d, d, false);
  switch (g % 4) {
    case TE_QKV: return make_geom(g, 3 * d, d, false);
    case TE_O: return make_geom(g, d, d, false);
    case TE_FFN1: return make_geom(g, f, d, false);
    default: return make_geom(g, d, f, false);
  }
}

// ------------------------------------------------------------------------------------------
// set-up, weight stream, tear-down
// ------------------------------------------------------------------------------------------

// Every thread.  ring = slots that fit; kind = the phase sequence this kernel runs; maps = its
// tensor maps (kernel parameters).
template <typename W>
__device__ void tc_setup(const Dims& D, int kind, int ring, const CUtensorMap* maps) {
  TcState& s = smem_tc<W>();
  for (int g = threadIdx.x; g < gemm_phase_count(D, kind); g += kThreads)
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(maps + g)) : "memory");
  const int n_g = gemm_phase_count(D, kind);
  const int grid = (int)gridDim.x;
  for (int g = threadIdx.x; g < n_g; g += kThreads) {        // one phase per thread
    const Geom G = gemm_geom(D, kind, g);
    PInfo& in = s.info[g];
    in.N = G.N;
    in.items = G.items;
    in.S = (unsigned char)G.S;
    in.kbs = (unsigned char)(G.KS / kKBlock);
    in.rtmax = (unsigned char)(G.RC / kRowTile);
  }
  __syncthreads();
  if (threadIdx.x == 0) {          // rotation: phase g starts at CTA (items of phases < g) % grid
    int off = 0;
    for (int g = 0; g < n_g; ++g) {
      s.info[g].first = (short)off;           // the offset, for now
      off += s.info[g].items;
      while (off >= grid) off -= grid;
    }
  }
  __syncthreads();
  for (int g = threadIdx.x; g < n_g; g += kThreads) {
    PInfo& in = s.info[g];
    int first = (int)blockIdx.x - in.first;
    if (first < 0) first += grid;
    in.first = (short)first;
    in.nj0 = (short)(first < in.items ? (in.items - first + grid - 1) / grid : 0);
  }
  if (threadIdx.x == 0) {
    for (int i = 0; i < kRingMax; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], 1);
    }
    mbar_init(&s.acc, 1);
    int sh = 0;
    while ((2 << sh) <= ring) ++sh;
    s.ring = 1 << sh;
    s.ring_sh = sh;
    s.kind = kind;
    s.n_g = n_g;
    s.p_g = 0; s.p_j = 0; s.p_kb = 0; s.p_seq = 0; s.p_M = 0; s.p_open = 0; s.p_spec = 0;
    s.c_seq = 0; s.acc_n = 0; s.last = 0; s.err = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    fence_proxy_async_smem();
  }
  if (threadIdx.x < 32) tmem_alloc(&s.tmem, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
}

// Thread 0: issue TMA loads of the CTA's next weight K-blocks while slots are free.  The
// cursor walks (phase, unit, K-block) over the GEMM phases of the current pass (p_M rows); with
// p_open it goes on past the pass's phase list into the next pass, speculating that it has the
// same rows (p_spec; tc_begin_pass drops those blocks if not).  With p_M = 0 (rows unknown) it
// stops after the chunk-0 units of phase 0.  block = wait for a free slot instead of returning
// when none is free.
template <typename W>
__device__ void tc_produce(const Dims& D, const CUtensorMap* maps, unsigned char* ring,
                           bool block) {
  TcState& s = smem_tc<W>();
  // the cursor in registers (the asm statements below clobber memory, which would make the
  // compiler reload every shared field after each of them)
  int g = s.p_g, j = s.p_j, kb = s.p_kb, seq = s.p_seq, M = s.p_M;
  int open = s.p_open, spec = s.p_spec;
  const int n_g = s.n_g, rsh = s.ring_sh, rmask = (1 << rsh) - 1;
  const int grid = (int)gridDim.x;
  PInfo in = g < n_g ? s.info[g] : PInfo{};
  int nj = g < n_g ? (M > 0 ? (int)s.pj[g] : (int)in.nj0) : 0;
  while (g < n_g) {
    if (j >= nj) {                               // next phase
      // between passes the row count is unknown: which units this CTA has depends on it past
      // the chunk-0 units of phase 0, so the stream waits there
      if (M == 0) break;
      g += 1; j = 0; kb = 0;
      if (g >= n_g) {
        if (!open) break;
        g = 0; open = 0; spec = 1;               // wrap to the next pass (same rows, presumed)
      }
      in = s.info[g];
      nj = M > 0 ? (int)s.pj[g] : (int)in.nj0;
      continue;
    }
    const int slot = seq & rmask, use = seq >> rsh;
    if (use > 0) {
      if (block) {
        if (!mbar_wait(&s.empty[slot], (use - 1) & 1, &s.err)) break;
      } else if (!mbar_test(&s.empty[slot], (use - 1) & 1)) {
        break;
      }
    }
    const int u = in.first + j * grid;
    const int item = u % in.items;
    const int tile = in.S == 1 ? item : item / in.S, sp = in.S == 1 ? 0 : item - tile * in.S;
    mbar_expect_tx(&s.full[slot], kSlotBytes);
    tma_load_2d(ring + (size_t)slot * kSlotBytes, maps + g, &s.full[slot],
                (sp * in.kbs + kb) * kKBlock, tile * kTileN);
    seq += 1;
    if (++kb == in.kbs) { kb = 0; ++j; }
    if (block) break;
  }
  s.p_g = g; s.p_j = j; s.p_kb = kb; s.p_seq = seq; s.p_M = M;
  s.p_open = open; s.p_spec = spec;
}

// Thread 0, at the start of a pass of M rows (pass_open: keep streaming into the next pass).
// Every block of the previous pass has been consumed.  If the stream went on into this pass
// presuming other rows, its blocks are dropped: each load is awaited (bounded) and its slot
// released as its MMAs would have, and the cursor restarts at this pass's first block.
template <typename W>
__device__ __forceinline__ void tc_begin_pass(int M, bool pass_open) {
  TcState& s = smem_tc<W>();
  if (!s.p_spec || s.p_M != M) {
    for (int q = s.c_seq; q < s.p_seq; ++q) {
      const int slot = q & (s.ring - 1);
      (void)mbar_wait(&s.full[slot], (q >> s.ring_sh) & 1, &s.err);
      mbar_arrive(&s.empty[slot]);
    }
    s.c_seq = s.p_seq;
    s.p_g = 0; s.p_j = 0; s.p_kb = 0;
  }
  s.p_spec = 0;
  s.p_M = M;
  s.p_open = pass_open ? 1 : 0;
}

// Every thread, at the start of a pass of M rows (after tc_begin_pass, before the barrier that
// precedes the pass's first phase): this CTA's units and chunk size of every GEMM phase.
template <typename W>
__device__ __forceinline__ void tc_plan(int M) {
  TcState& s = smem_tc<W>();
  for (int g = threadIdx.x; g < s.n_g; g += kThreads) {
    int rc, nch, nj;
    tc_chunks(s.info[g], M, (int)gridDim.x, rc, nch, nj);
    s.pj[g] = (short)nj;
    s.prt[g] = (unsigned char)(rc / kRowTile);
  }
}

// Every thread, at the end of the kernel: wait (bounded) for the weight loads still in flight
// and for the tensor cores, then free the tensor memory.
template <typename W>
__device__ void tc_teardown() {
  TcState& s = smem_tc<W>();
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int q = s.c_seq; q < s.p_seq; ++q)
      (void)mbar_wait(&s.full[q & (s.ring - 1)], (q >> s.ring_sh) & 1, &s.err, 1000000000ull);
    mma_commit(&s.acc);
    (void)mbar_wait(&s.acc, s.acc_n & 1, &s.err, 1000000000ull);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (threadIdx.x < 32) tmem_dealloc(s.tmem, kTmemCols);
}

// ------------------------------------------------------------------------------------------
// B staging
// ------------------------------------------------------------------------------------------

__device__ __forceinline__ void put4_b(unsigned char* bb, int r, int kk, int rtiles, float4 v) {
  __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
  uint2 u;
  u.x = *reinterpret_cast<unsigned*>(&a);
  u.y = *reinterpret_cast<unsigned*>(&b);
  *reinterpret_cast<uint2*>(bb + b_offset(r, kk, rtiles)) = u;
}

// Stage rows m0..m0+mt of the GEMM input, K elements k0..k0+KS, into the B layout (rows mt..
// rtiles*16 zero).  LayerNorm / embedding rows are computed whole (the statistics need the
// full row); `store` writes the full normalised fp32 rows to g.x_store.  lnv: shared memory for
// the phase's LayerNorm vectors (4 K elements of W).
template <typename W>
__device__ __noinline__ void stage_b(const GemmArgs<W>& g, const EmbedTabs<W>& T, const Dims& D, int m0,
                        int mt, int k0, int KS, int rtiles, bool store, unsigned char* bb,
                        W* lnv) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int K = g.K;
  // zero rows mt .. rtiles*16 - 1 (16-byte stores)
  const int zrows = rtiles * kRowTile - mt;
  if (zrows > 0) {
    const int per_row = KS / 8;
    for (int f = threadIdx.x; f < zrows * per_row; f += kThreads) {
      const int r = mt + f / per_row, kk = (f % per_row) * 8;
      *reinterpret_cast<uint4*>(bb + b_offset(r, kk, rtiles)) = make_uint4(0u, 0u, 0u, 0u);
    }
  }
  const bool any_ln = g.ln_a_g != nullptr || g.ln_b_g != nullptr || g.emb_tok != nullptr;
  if (!any_ln) {
    const bool wsrc = g.xw_src != nullptr;
    const int E = wsrc ? 8 : 4;                  // elements per 16-byte load
    const int KE = KS / E, F = mt * KE;
    for (int f0 = 0; f0 < F; f0 += kThreads * kStageB) {
      uint4 v[kStageB];
#pragma unroll
      for (int j = 0; j < kStageB; ++j) {
        const int f = f0 + j * kThreads + (int)threadIdx.x;
        if (f < F) {
          const int r = f / KE, kk = (f - r * KE) * E;
          v[j] = wsrc ? ld_act16(g.xw_src + (size_t)(m0 + r) * K + k0 + kk)
                      : ld_act16(g.x_src + (size_t)(m0 + r) * K + k0 + kk);
        }
      }
#pragma unroll
      for (int j = 0; j < kStageB; ++j) {
        const int f = f0 + j * kThreads + (int)threadIdx.x;
        if (f < F) {
          const int r = f / KE, kk = (f - r * KE) * E;
          if (wsrc) {
            *reinterpret_cast<uint4*>(bb + b_offset(r, kk, rtiles)) = v[j];
          } else {
            const float4 x = make_float4(__uint_as_float(v[j].x), __uint_as_float(v[j].y),
                                         __uint_as_float(v[j].z), __uint_as_float(v[j].w));
            if (store) *reinterpret_cast<float4*>(g.x_store + (size_t)(m0 + r) * K + k0 + kk) = x;
            put4_b(bb, r, kk, rtiles, x);
          }
        }
      }
    }
    return;
  }
  // the LayerNorm vectors of this phase (identical for every row) into shared memory once:
  // lnv = [ln_a gamma | ln_a beta | ln_b gamma | ln_b beta], K elements each, in W
  const W *ga_g = g.ln_a_g, *ga_b = g.ln_a_b, *gb_g = g.ln_b_g, *gb_b = g.ln_b_b;
  if (lnv != nullptr) {
    const W* src[4] = {g.ln_a_g, g.ln_a_b, g.ln_b_g, g.ln_b_b};
    const int per = K * (int)sizeof(W) / 16;              // 16-byte chunks per vector
    for (int f = threadIdx.x; f < 4 * per; f += kThreads) {
      const int v = f / per, c = f - v * per;
      if (src[v] != nullptr)
        *reinterpret_cast<uint4*>(reinterpret_cast<char*>(lnv + (size_t)v * K) + c * 16) =
            ldg_nc_v4(reinterpret_cast<const char*>(src[v]) + c * 16);
    }
    __syncthreads();
    if (ga_g != nullptr) { ga_g = lnv; ga_b = lnv + K; }
    if (gb_g != nullptr) { gb_g = lnv + 2 * K; gb_b = lnv + 3 * K; }
  }
  // each warp takes two rows at a time (both rows' loads issued before either is normalised)
  const int nI = K / 128;
  for (int r0 = warp; r0 < mt; r0 += 2 * kWarps) {
    float4 v[2][kMaxRowRegs];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int r = r0 + h * kWarps;
      if (r >= mt) break;
      const int m = m0 + r;
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
            v[h][i] = make_float4(e.x * D.emb_scale + ps.x, e.y * D.emb_scale + ps.y,
                                  e.z * D.emb_scale + ps.z, e.w * D.emb_scale + ps.w);
          }
        }
      } else {
        const float* src = g.x_src + (size_t)m * K;
#pragma unroll
        for (int i = 0; i < kMaxRowRegs; ++i)
          if (i < nI) v[h][i] = *reinterpret_cast<const float4*>(src + lane * 4 + 128 * i);
      }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int r = r0 + h * kWarps;
      if (r >= mt) break;
      const int m = m0 + r;
      if (ga_g != nullptr) ln_regs(v[h], nI, K, ga_g, ga_b, D.eps);
      if (store && g.x_store != nullptr) {
#pragma unroll
        for (int i = 0; i < kMaxRowRegs; ++i)
          if (i < nI)
            *reinterpret_cast<float4*>(g.x_store + (size_t)m * K + lane * 4 + 128 * i) = v[h][i];
      }
      if (gb_g != nullptr) ln_regs(v[h], nI, K, gb_g, gb_b, D.eps);
#pragma unroll
      for (int i = 0; i < kMaxRowRegs; ++i) {
        const int k = lane * 4 + 128 * i;
        if (i < nI && k >= k0 && k < k0 + KS) put4_b(bb, r, k - k0, rtiles, v[h][i]);
      }
    }
  }
}

// ------------------------------------------------------------------------------------------
// the GEMM phase
// ------------------------------------------------------------------------------------------

// Element epilogue of output (m, n) with value v = accumulated dot product (+ nothing else).
template <typename W>
__device__ __forceinline__ void epi_store(const GemmArgs<W>& g, const Dims& D, int m, int n,
                                          float v, float bias, float resid) {
  v += bias;
  switch (g.epi) {
    case EPI_STORE: g.out[(size_t)m * g.ld + n] = v; break;
    case EPI_ACT: g.out_w[(size_t)m * g.ld + n] = from_f<W>(act_fn(v, D.act)); break;
    case EPI_RESID: g.out[(size_t)m * g.ld + n] = v + resid; break;
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
    case EPI_LOGITS: g.out[(size_t)m * g.ld + n] = v; break;
    default: break;
  }
}

// The accumulated values of lane quadrant q (this warp's, q = warp % 4) for the 16-row tile rt:
// the naccs accumulators summed in a fixed order (v[r] = row 16 rt + r).
__device__ __forceinline__ void tc_load_acc(uint32_t tmem, int q, int rt, int naccs,
                                            float (&v)[16]) {
  const uint32_t ta = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(rt * kRowTile);
  tmem_ld16(ta, v);
  for (int c = 1; c < naccs; ++c) {
    float w[16];
    tmem_ld16(ta + (uint32_t)(c * kMaxChunk), w);
#pragma unroll
    for (int r = 0; r < 16; ++r) v[r] += w[r];
  }
}

// Thread 0: the MMAs of one item over rtiles 16-row tiles.  K-block kb accumulates into
// accumulator kb % kAccs (tensor-memory columns (kb % kAccs) * kMaxChunk + 16 rt ..), so that
// kAccs dependent chains of MMAs run side by side; within a chain the K-blocks and the K = 16
// steps are in ascending order.  Every K-block's slot is released by a commit once its MMAs
// are done (the stream is topped up after the item, while the CTA waits at barriers, and on
// demand when a block has not been issued yet).  Returns false if a wait failed.
template <typename W>
__device__ __forceinline__ bool tc_issue_item(const Dims& D, const CUtensorMap* maps,
                                              unsigned char* ring, unsigned char* bb, int kbs,
                                              int rtiles) {
  TcState& s = smem_tc<W>();
  const uint32_t idesc = idesc_bf16(kTileN, kRowTile * rtiles);
  const uint32_t bbase = smem_u32(bb);
  const uint32_t tmem = s.tmem;
  const int rmask = s.ring - 1, rsh = s.ring_sh;
  const uint32_t rbase = smem_u32(ring);
  int cseq = s.c_seq;
  bool ok = true;
  tc_fence_after();
  for (int kb = 0; kb < kbs && ok; ++kb) {
    while (s.p_seq <= cseq) {
      const int before = s.p_seq;
      tc_produce<W>(D, maps, ring, true);
      if (s.err) { ok = false; break; }
      if (s.p_seq == before) { s.err = 2; ok = false; break; }   // the stream cannot supply it
    }
    if (!ok) break;
    const int slot = cseq & rmask, use = cseq >> rsh;
    if (!mbar_wait(&s.full[slot], use & 1, &s.err)) { ok = false; break; }
    tc_fence_after();
    // descriptors advance by 32 bytes (2 in the start-address field) per K = 16 step
    const uint64_t a0 = sw128_desc(rbase + (uint32_t)(slot * kSlotBytes));
    const uint32_t col = (uint32_t)((kb % kAccs) * kMaxChunk);
    // one MMA covers every 16-row tile of the chunk (N = 16 rtiles): the B rows of a K-block
    // are contiguous, 128 bytes apart, and the accumulator columns of the tiles adjacent
    const uint64_t b0 = sw128_desc(bbase + (uint32_t)(kb * rtiles * 2048));
#pragma unroll
    for (int k16 = 0; k16 < kKBlock / 16; ++k16)
      mma_bf16(tmem + col, a0 + (uint64_t)(2 * k16), b0 + (uint64_t)(2 * k16), idesc,
               (kb >= kAccs || k16 > 0) ? 1u : 0u);
    mma_commit(&s.empty[slot]);
    cseq += 1;
  }
  s.c_seq = cseq;
  return ok;
}

// GEMM phase g of the current phase sequence over the M rows of ga, on the tensor cores.
// Every thread of every CTA calls it (CTAs without items of the phase only keep the weight
// stream going and, for the LM head, publish empty argmax partials).  Returns false if a
// bounded wait gave up.
template <typename W>
__device__ __noinline__ bool tc_gemm_phase(const GemmArgs<W>& ga, const EmbedTabs<W>& T,
                                           const Dims& D, int gph, const CUtensorMap* maps,
                                           unsigned char* ring, unsigned char* bb, float* epi,
                                           Partial* rowp, float* red, unsigned* cnt) {
  TcState& s = smem_tc<W>();
  const PInfo in = s.info[gph];
  const int S = in.S, kbs = in.kbs, KS = kbs * kKBlock, N = in.N;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int M = ga.M;
  const int grid = (int)gridDim.x;
  const int RC = (int)s.prt[gph] * kRowTile, nj = s.pj[gph];
  const bool argmax = ga.epi == EPI_ARGMAX;
  const int naccs = kbs < kAccs ? kbs : kAccs;
  if (argmax)             // the CTA's running argmax partial of every row of the pass
    for (int m = threadIdx.x; m < M; m += kThreads) rowp[m] = Partial{-INFINITY, 0x7fffffff, 0.f, 0};
  if (nj == 0) {
    if (argmax)
      for (int m = threadIdx.x; m < M; m += kThreads)
        ga.part[(size_t)blockIdx.x * ga.part_ld + m] = Partial{-INFINITY, 0x7fffffff, 0.f, 0};
    if (threadIdx.x == 0) tc_produce<W>(D, maps, ring, false);
    return true;
  }
  int staged_key = -1;
  for (int j = 0; j < nj; ++j) {
    {
      const int u = in.first + j * grid;
      const int item = u % in.items, ch = u / in.items;
      const int tile = S == 1 ? item : item / S, sp = S == 1 ? 0 : item - tile * S;
      const int m0 = ch * RC, mt = M - m0 < RC ? M - m0 : RC;
      const int rtiles = (mt + kRowTile - 1) / kRowTile;
      const int n0 = tile * kTileN;
      // stage the B operand (rows of this chunk, the unit's K-slice) when it changes; the CTA
      // holding item 0 of a chunk stores the chunk's normalised rows (x_store)
      const int key = ch * S + sp;
      if (key != staged_key) {
        __syncthreads();                           // the previous MMAs are done (acc wait)
        stage_b<W>(ga, T, D, m0, mt, sp * KS, KS, rtiles, item == 0, bb,
                   reinterpret_cast<W*>(epi));
        fence_proxy_async_smem();
        __syncthreads();
        staged_key = key;
      }
      // epilogue operands that do not depend on this phase's products: the bias of this
      // thread's feature (f for the shared-memory path, nfq for the warp-parallel one)
      const int f = threadIdx.x % kTileN;
      const int nf = n0 + f;
      const int q = warp & 3, nfq = n0 + 32 * q + lane;
      const float bias = (ga.bias != nullptr && nf < N) ? to_f(ga.bias[nf]) : 0.f;
      const float bq = (ga.bias != nullptr && nfq < N) ? to_f(ga.bias[nfq]) : 0.f;
      if (threadIdx.x == 0) {
        (void)tc_issue_item<W>(D, maps, ring, bb, kbs, rtiles);
        mma_commit(&s.acc);
        (void)mbar_wait(&s.acc, s.acc_n & 1, &s.err);
        if (!s.err) tc_produce<W>(D, maps, ring, false);   // slots released: stream on
      }
      __syncthreads();
      if (s.err) return false;
      tc_fence_after();
      if (!argmax) {
        // straight from tensor memory: warp w owns lane quadrant q = w % 4 (features n0 + 32 q
        // + lane) of the 16-row tiles w / 4, w / 4 + 3, ...; the accumulators are summed in a
        // fixed order; one thread per feature, so every row's stores are coalesced
        const size_t rs = (size_t)D.rows;
        if (S > 1) {
          // split K: publish this slice's partial; the last of the S CTAs to arrive for this
          // tile and chunk sums the slices in ascending order and runs the epilogue
          for (int rt = warp >> 2; rt < rtiles; rt += kWarps / 4) {
            float v[16];
            tc_load_acc(s.tmem, q, rt, naccs, v);
            const int rows = mt - rt * kRowTile < kRowTile ? mt - rt * kRowTile : kRowTile;
            if (nfq < N)
              for (int r = 0; r < rows; ++r)
                red[((size_t)sp * rs + m0 + rt * kRowTile + r) * N + nfq] = v[r];
          }
          __threadfence();
          __syncthreads();
          if (threadIdx.x == 0) {
            unsigned* c = cnt + (size_t)(tile * ((D.rows + kRowTile - 1) / kRowTile) +
                                         m0 / kRowTile) % kCounterSlots;
            const unsigned old = atomicAdd(c, 1u);
            s.last = old == (unsigned)(S - 1);
            if (s.last) atomicExch(c, 0u);
          }
          __syncthreads();
          if (s.last) {
            __threadfence();
            for (int rt = warp >> 2; rt < rtiles; rt += kWarps / 4) {
              const int rows = mt - rt * kRowTile < kRowTile ? mt - rt * kRowTile : kRowTile;
              if (nfq < N)
                for (int r = 0; r < rows; ++r) {
                  const int m = m0 + rt * kRowTile + r;
                  float acc = 0.f;
                  for (int qq = 0; qq < S; ++qq) acc += __ldcg(red + ((size_t)qq * rs + m) * N + nfq);
                  const float resid = ga.epi == EPI_RESID ? ga.resid[(size_t)m * ga.ld + nfq] : 0.f;
                  epi_store<W>(ga, D, m, nfq, acc, bq, resid);
                }
            }
          }
        } else {
          for (int rt = warp >> 2; rt < rtiles; rt += kWarps / 4) {
            float v[16];
            tc_load_acc(s.tmem, q, rt, naccs, v);
            const int rows = mt - rt * kRowTile < kRowTile ? mt - rt * kRowTile : kRowTile;
            if (nfq < N)
#pragma unroll
              for (int r = 0; r < 16; ++r) {
                if (r < rows) {
                  const int m = m0 + rt * kRowTile + r;
                  const float resid = ga.epi == EPI_RESID ? ga.resid[(size_t)m * ga.ld + nfq] : 0.f;
                  epi_store<W>(ga, D, m, nfq, v[r], bq, resid);
                }
              }
          }
        }
      } else {
        // LM head argmax: the tile goes through shared memory, one 16-row tile at a time
        for (int rt = 0; rt < rtiles; ++rt) {
          const int rows = mt - rt * kRowTile < kRowTile ? mt - rt * kRowTile : kRowTile;
          if (warp < 4) {
            float v[16];
            tc_load_acc(s.tmem, warp, rt, naccs, v);
#pragma unroll
            for (int r = 0; r < 16; ++r) epi[r * kEpiLd + warp * 32 + lane] = v[r];
          }
          __syncthreads();
          // row r of the tile -> warp r % 12; lane l takes features l, l + 32, l + 64, l + 96,
          // the lanes' partials meet in a fixed butterfly, and lane 0 merges the item's partial
          // into the row's running one (items in ascending order)
          for (int r = warp; r < rows; r += kWarps) {
            Partial a{-INFINITY, 0x7fffffff, 0.f, 0};
#pragma unroll
            for (int qq = 0; qq < 4; ++qq) {
              const int ff = lane + 32 * qq, n = n0 + ff;
              if (n < N) argmax_push(epi[r * kEpiLd + ff], n, a.mx, a.idx, a.sum, a.nan);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) partial_merge(a, shfl_partial(a, o));
            if (lane == 0) partial_merge(rowp[m0 + rt * kRowTile + r], a);
          }
          __syncthreads();
        }
      }
      (void)bias;
      tc_fence_before();
      __syncthreads();
      if (threadIdx.x == 0) s.acc_n += 1;
    }
  }
  if (argmax) {
    __syncthreads();
    for (int m = threadIdx.x; m < M; m += kThreads)
      ga.part[(size_t)blockIdx.x * ga.part_ld + m] = rowp[m];
  }
  __syncthreads();
  return true;
}

}  // namespace pd

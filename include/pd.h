/*
 * pd.h — C ABI of a single-GPU (GB300, sm_103a) parallel decoder for encoder-decoder
 * translation transformers, after "Accelerating Transformer Inference for Translation via
 * Parallel Decoding" (Santilli et al., arXiv 2305.10427).
 *
 * The paper states the problem as: given a source sentence x = (x_1..x_n), return
 * y = (y_1..y_m) with y_i = argmax p_theta(y_i | y_1..y_{i-1}, x) (Section 3.1, Eq. 1-2),
 * and solves that triangular system (Eq. 3-4) with Jacobi (Algorithm 1), GS-Jacobi
 * (Algorithm 2) or Hybrid GS-Jacobi (Algorithm 3) fixed-point iterations, drafts initialised
 * to PAD (Section 3.3, InitT) and stopped when a block no longer changes (Eq. 5, StopC).
 *
 * Conventions for every entry point:
 *  - Host pointers are plain CPU memory owned by the caller; "d_" pointers are device memory
 *    of the context's GPU owned by the caller.  The library never keeps a caller pointer.
 *  - The library allocates all of its device memory in pd_create, sized for the capacities in
 *    pd_config; pd_encode / pd_decode allocate nothing (pd_debug_logits is the one exception,
 *    a test-only call).
 *  - Arguments are checked before anything is launched; a bad argument returns PD_EINVAL and
 *    leaves the context unchanged.  A CUDA failure returns PD_ECUDA.  pd_last_error() gives a
 *    one-line reason for the last failure on that context.  No C++ exception crosses the ABI.
 *  - A context is used by one host thread at a time.  All work is issued on the context's
 *    stream (the one passed to pd_create, or a stream the library creates).
 */
#ifndef PD_H
#define PD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  PD_OK = 0,
  PD_EINVAL = -1,    /* bad argument or unsupported configuration */
  PD_ENOMEM = -2,    /* device allocation failed in pd_create */
  PD_ECUDA = -3,     /* a CUDA runtime call or kernel failed */
  PD_ENOTCONV = -4,  /* the pass budget (pd_decode_params.max_passes) ran out first */
  PD_ENAN = -5,      /* a NaN appeared in the logits */
  PD_ESTATE = -6,    /* pd_decode before any successful pd_encode */
  PD_ETIMEOUT = -7   /* a device-side wait gave up (the kernel returned instead of hanging) */
} pd_status;

typedef enum {
  PD_GREEDY = 0,            /* Eq. 2: one position per decoder pass */
  PD_JACOBI = 1,            /* Algorithm 1: the whole sentence is one block */
  PD_GS_JACOBI = 2,         /* Algorithm 2: blocks of b positions, solved in order */
  PD_HYBRID_GS_JACOBI = 3   /* Algorithm 3: GS-Jacobi up to h, EOS exit, greedy tail */
} pd_method;

typedef enum { PD_ACT_RELU = 0, PD_ACT_SILU = 1, PD_ACT_GELU = 2 } pd_activation;
typedef enum { PD_DTYPE_F32 = 0, PD_DTYPE_BF16 = 1 } pd_dtype;

/* Model structure and capacities.  The paper runs a base (d=512, 6+6 layers) and a big
 * (d=1024, 12+12 layers) transformer (Section 4.1, "Model Configuration"); everything it
 * leaves to the model library is fixed here: token embedding scaled by sqrt(d_model) and
 * tied with the output projection (no logits bias), sinusoidal ([sin | cos], frequency
 * 10000^(-2k/d), from position 0) or learned positions, post-LN (x = LN(x + f(x))) or pre-LN
 * (x = x + f(LN(x)) with embedding and final LayerNorms), attention scale 1/sqrt(d_head).
 * Supported: d_model and d_ff multiples of 256, d_model / n_heads in {32, 64, 128},
 * n_enc_layers and n_dec_layers in [1, 16]. */
typedef struct {
  int d_model, n_heads, d_ff, n_enc_layers, n_dec_layers, vocab;
  int activation;    /* pd_activation */
  int pre_ln;        /* 0: post-LN, 1: pre-LN */
  int learned_pos;   /* 0: sinusoidal, 1: learned table of max_pos rows */
  int max_pos;       /* rows of the learned position table */
  int dtype;         /* pd_dtype: storage of every parameter; activations are fp32 */
  int pad_id, eos_id, bos_id;
  float ln_eps;
  int max_src_len;   /* capacity: longest source sentence pd_encode accepts */
  int max_tgt_len;   /* capacity: largest max_len pd_decode accepts */
  int max_batch;     /* capacity: sentences one pd_encode_batch / pd_decode_batch carries,
                        0 or 1..64 (0 = 1); each needs its own key/value caches */
  int gemm_engine;   /* pd_gemm_engine: how the decoder passes run (fp32: SIMT or CLUSTER) */
  int seed;          /* pd_create with weights = NULL: the seed of the drawn weights */
  int kv_pages;      /* capacity of each decoder layer's self-attention key/value pool, in
                        pages of 16 positions (0 = max_batch * ceil(max_tgt_len / 16)); a
                        decode needs sum over its sentences of ceil(max_len / 16) pages */
  int cluster_size;  /* PD_ENGINE_CLUSTER: CTAs per thread-block cluster, 1, 2, 4 or 8 (0 = 8;
                        1 = a plain cooperative launch, every CTA a cluster of one) */
} pd_config;

/* How a context runs its decoder passes (and the matrix products of its encoder).  Every pass
 * of a context uses the same engine, so each row's arithmetic is the same whatever the pass
 * carries and every decoding method returns exactly the context's greedy tokens; the engines
 * round differently (all within the parity bar).
 *  PD_ENGINE_SIMT: CUDA-core dot products spread over every SM, the 8 steps of a decoder layer
 *    separated by grid barriers.
 *  PD_ENGINE_TENSOR (bf16 only): the SIMT engine's phases with every matrix product on the
 *    5th-generation tensor cores (tcgen05, accumulators in tensor memory), weight tiles
 *    streamed by TMA.
 *  PD_ENGINE_CLUSTER: a decoder layer as three super-phases (self-attention, cross-attention,
 *    FFN), each run per attention head or per slice of FFN hidden units by a thread-block
 *    cluster of cluster_size CTAs that exchange rows through distributed shared memory, with
 *    one grid barrier per super-phase; CUDA-core products, SIMT encoder.
 *  PD_ENGINE_AUTO: SIMT. */
typedef enum {
  PD_ENGINE_AUTO = 0,
  PD_ENGINE_SIMT = 1,
  PD_ENGINE_TENSOR = 2,
  PD_ENGINE_CLUSTER = 3
} pd_gemm_engine;

typedef struct pd_ctx pd_ctx;

/* Size in bytes of the weight blob for cfg: every parameter in the documented order (token
 * embedding [V,d]; learned positions [max_pos,d] if any; pre-LN only: encoder and decoder
 * embedding-LN and final-LN gain/bias; then per encoder layer wqkv [3d,d], bqkv, wo [d,d],
 * bo, ln1 g/b, w1 [f,d], b1, w2 [d,f], b2, ln2 g/b; then per decoder layer wqkv, bqkv, wo, bo,
 * ln1 g/b, wq_c [d,d], bq_c, wkv_c [2d,d], bkv_c, wo_c [d,d], bo_c, ln2 g/b, w1, b1, w2, b2,
 * ln3 g/b), row-major, linear maps stored [out, in], elements float32 or bfloat16 bits.
 * Returns 0 for an invalid cfg. */
size_t pd_weights_nbytes(const pd_config* cfg);

/* Create a context on the current CUDA device: validate cfg, allocate every device buffer for
 * the capacities in cfg, and upload the weight blob (host memory, nbytes =
 * pd_weights_nbytes(cfg)).  With weights = NULL and nbytes = 0 the library draws the weights
 * itself from cfg->seed: element e of the blob's tensor number k (blob order, from 0) is
 * 0.02 z, z the Box-Muller normal of the first two words of Philox-4x32-10 (Salmon et al., SC
 * 2011) at counter (e / 2, k, 0, 0), key (seed, 0x5EED5EED) (cosine for even e, sine for odd),
 * LayerNorm gains 1 and biases 0, rounded to the parameter type; pd_export_weights returns
 * them.  stream is a cudaStream_t (NULL: the library creates its own).  On success *out owns
 * all device memory until pd_destroy. */
pd_status pd_create(const pd_config* cfg, const void* weights, size_t nbytes, void* stream,
                    pd_ctx** out);

/* Copy the device weights back in blob order (dst host memory of nbytes). */
pd_status pd_export_weights(pd_ctx* ctx, void* dst, size_t nbytes);

/* Run the encoder once for a source sentence x_1..x_n (host int32 ids, 1 <= n_src <=
 * max_src_len, each in [0, vocab)) and cache the cross-attention keys and values of every
 * decoder layer; only the decoder runs per iteration (Fig. 1; Section 4.1 caches keys and
 * values).  Synchronous. */
pd_status pd_encode(pd_ctx* ctx, const int32_t* src, int n_src);

/* As pd_encode, with the ids already in device memory (d_src); asynchronous on the context
 * stream (ids are not range-checked; out-of-range ids are clamped on the device). */
pd_status pd_encode_device(pd_ctx* ctx, const int32_t* d_src, int n_src);

/* When a block's repeated passes end.  Both rules return the same tokens (after k passes the
 * first k block positions are exact, Section 3.4, Proposition 1); they differ in passes.
 *  PD_STOP_UNCHANGED: StopC of Eq. 5 (Section 3.3): the block ends when a pass leaves all of
 *    its tokens unchanged, or after as many passes as the block has positions.
 *  PD_STOP_PREFIX: also ends the block once the leading unchanged count c of a pass reaches
 *    blk - 1: the first c + 1 new tokens are then exact (each was predicted from inputs
 *    already equal to the solution), so the whole block is, and the confirming pass that
 *    Eq. 5 needs is skipped.  The paper leaves other stopping conditions to future work
 *    (Section 5, Conclusions); this is one, with the same result and at most as many passes. */
typedef enum { PD_STOP_UNCHANGED = 0, PD_STOP_PREFIX = 1, PD_STOP_SUFFIX = 2 } pd_stop_rule;

/* PD_STOP_SUFFIX: the accepted-prefix rule, with each further pass of a block re-running only
 * the block positions after its exact prefix (the first c + 1 new tokens of the last pass):
 * the same tokens, passes and trace as PD_STOP_PREFIX (the rows it skips would reproduce their
 * tokens bit for bit), fewer rows per pass.  The paper names other stopping conditions and
 * cheaper iterations as future work (Section 5). */

/* The drafts a new block of Jacobi / GS-Jacobi / Hybrid GS-Jacobi starts from (InitT,
 * Section 3.3).  PD_INIT_PAD: every draft is PAD, as in the paper.  PD_INIT_LAST: every draft
 * is the last token already decided, y_{i-1} (one of the other initialisations the paper
 * leaves to future work, Section 5).  Proposition 1 holds for any initialisation: the tokens are
 * the greedy ones either way; the pass counts differ. */
typedef enum { PD_INIT_PAD = 0, PD_INIT_LAST = 1 } pd_init_rule;

typedef struct {
  int method;       /* pd_method */
  int b;            /* block size for GS-Jacobi / hybrid (>= 1); ignored by greedy, jacobi */
  int max_len;      /* 1 <= max_len <= max_tgt_len; for jacobi / gs_jacobi it is the known
                       target length m of Section 4.1 */
  int h;            /* hybrid: parallel part up to position h (0 = max_len) */
  int stop_at_eos;  /* greedy / jacobi / gs_jacobi: end the returned y at the first EOS */
  int max_passes;   /* 0 = no limit; else stop with PD_ENOTCONV after this many passes */
  int stop_rule;    /* pd_stop_rule (0 = Eq. 5) */
  int init;         /* pd_init_rule (0 = PAD, the paper's InitT) */
} pd_decode_params;

/* One decoder pass of the trace (DDGviz-style, Section 3.5): pass number (1-based), block
 * start position i (1-based), block length, number of leading block positions whose new
 * token equals the previous draft, StopC (Eq. 5) flag (under any stop rule), index of the
 * first EOS in the new block tokens (-1 if none), rows the pass computed (block_len, or fewer
 * under PD_STOP_SUFFIX). */
typedef struct {
  int32_t step, block_start, block_len, n_converged, stop, eos_idx, n_rows;
} pd_trace_step;

/* Decode the sentence last given to pd_encode.  Outputs (host): y[0..*n_y) = y_1..y_m
 * (capacity max_len), *n_iters = decoder passes (encoder excluded).  Optional trace (NULL to
 * skip): trace[trace_cap], trace_tokens[trace_cap][max_len] (row t holds the pass's
 * block_len new tokens), trace_probs same shape (softmax probability of each argmax token);
 * *n_trace = rows written (min(passes, trace_cap)).  Synchronous.  Returns PD_ESTATE without
 * a prior pd_encode. */
pd_status pd_decode(pd_ctx* ctx, const pd_decode_params* p, int32_t* y, int* n_y, int* n_iters,
                    pd_trace_step* trace, int32_t* trace_tokens, float* trace_probs,
                    int trace_cap, int* n_trace);

/* As pd_decode, asynchronous on the context stream, outputs in device memory: d_y[max_len]
 * and d_info[4] = {n_y, n_iters, status, n_trace}.  Parameters are checked on the host. */
pd_status pd_decode_device(pd_ctx* ctx, const pd_decode_params* p, int32_t* d_y,
                           int32_t* d_info);

/* Batched serving (several independent sentences decoded together; the paper decodes one
 * sentence at a time, Section 4.1, and every result below is exactly that sentence's alone).
 *
 * pd_encode_batch: run the encoder for sentences s = 0..n_sent-1 (1 <= n_sent <= max_batch),
 * sentence s being src[offsets[s] .. offsets[s+1]) (host int32; offsets[0] = 0, every length in
 * [1, max_src_len], ids in [0, vocab)), caching each one's cross-attention keys and values in
 * slot s.  Synchronous.  pd_encode is pd_encode_batch of one sentence. */
pd_status pd_encode_batch(pd_ctx* ctx, const int32_t* src, const int32_t* offsets, int n_sent);

/* As pd_encode_batch with the ids in device memory (d_src) and offsets on the host;
 * asynchronous on the context stream (ids are not range-checked). */
pd_status pd_encode_batch_device(pd_ctx* ctx, const int32_t* d_src, const int32_t* offsets,
                                 int n_sent);

/* Decode the n_sent sentences of the last pd_encode_batch together: one decoder pass carries
 * the current block of every sentence that is not finished (at most 512 rows in all: the sum
 * over sentences of min(block size, max_len) must fit), each sentence with its own block
 * position, convergence test, EOS handling and pass count, as pd_decode would run it alone.
 * p gives the method and its parameters for all sentences; max_len (host int32[n_sent], or
 * NULL for p->max_len everywhere) the known length m of each.  Outputs (host): y[s * y_ld ..]
 * = sentence s's tokens (y_ld >= its max_len), n_y[s], n_iters[s] = passes in which sentence s
 * took part.  No trace.  Synchronous.  Returns PD_OK, or the status of the first sentence that
 * failed (outputs are filled for all). */
pd_status pd_decode_batch(pd_ctx* ctx, const pd_decode_params* p, int n_sent,
                          const int32_t* max_len, int32_t* y, int y_ld, int32_t* n_y,
                          int32_t* n_iters);

/* As pd_decode_batch, asynchronous on the context stream, outputs in device memory:
 * d_y[n_sent][y_ld] and d_info[n_sent][4] = {n_y, n_iters, status, n_trace}. */
pd_status pd_decode_batch_device(pd_ctx* ctx, const pd_decode_params* p, int n_sent,
                                 const int32_t* max_len, int32_t* d_y, int y_ld,
                                 int32_t* d_info);

/* Test-only: teacher-forced logits of one decoder pass over the input tokens y_in[0..len)
 * at positions 0..len-1 (row t scores position t+1, Eq. 1) for the sentence last encoded.
 * logits: host float32 [len][vocab].  Allocates a temporary device buffer; overwrites the
 * decoder's key/value cache.  Synchronous; PD_ETIMEOUT if a device wait gave up during the
 * pass (no logits are returned then). */
pd_status pd_debug_logits(pd_ctx* ctx, const int32_t* y_in, int len, float* logits);

/* Test-only, allocation-free variant of pd_debug_logits (the paper has no counterpart: this
 * is a service for callers that may not allocate device memory, e.g. a process whose device
 * memory is owned by another pool or that must not grow after start-up).  Same arguments and
 * results as pd_debug_logits, but the logits are staged in a fixed 4 MiB array inside the
 * library's device image instead of a per-call allocation, so len * vocab must not exceed
 * 1,048,576 (PD_EINVAL otherwise).  Every GPU that loads the library holds the array until the
 * process exits.  pd_create looks up the array's device address for its device (current while
 * it runs) and keeps it in the context, so this call does no set-up of its own.  All calls
 * share the one array, which keeps the last call's contents: calls that overlap on the GPU
 * (several contexts or threads at once) race and must be serialised by the caller.  Like
 * pd_debug_logits it overwrites the decoder's key/value cache and synchronises the context
 * stream; PD_ETIMEOUT if a device wait gave up during the pass.  Calls no device allocator. */
pd_status pd_debug_logits_static(pd_ctx* ctx, const int32_t* y_in, int len, float* logits);

/* Test-only failure-detection check (the paper has no counterpart).  Runs, on the context's
 * stream, one thread of the kernels' bounded device-side wait (the wait of the grid barriers)
 * against a counter that nothing advances, with a limit of limit_ns nanoseconds instead of the
 * kernels' 10 s.  The wait must give up: on return *status holds the status the device raised
 * (PD_ETIMEOUT expected), and the call returns PD_OK if the wait also raised its abort flag
 * (PD_ESTATE otherwise).  limit_ns in (0, 1e10]; PD_EINVAL otherwise.  Synchronous; allocates
 * and frees 16 bytes of device memory; the context stays usable. */
pd_status pd_debug_wait_timeout(pd_ctx* ctx, uint64_t limit_ns, int* status);

/* The context's cudaStream_t. */
void* pd_stream(pd_ctx* ctx);

/* Number of the library's kernel launches issued on this context so far. */
int64_t pd_launch_count(const pd_ctx* ctx);

/* One-line reason for the last failure on ctx ("" if none); valid until the next call.  With
 * ctx = NULL: the reason of the calling thread's last failed pd_create (which returns no
 * context to ask). */
const char* pd_last_error(const pd_ctx* ctx);

/* Free every device buffer and the context (NULL is a no-op). */
void pd_destroy(pd_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* PD_H */

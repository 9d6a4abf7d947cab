/*
 * tvl.h — C ABI of the GB300 batch-1 FP32 decode library (libtvl.so).
 *
 * The library runs the single-token decode step of a Llama-2-architecture
 * decoder on one GPU (sm_103a): every weight is streamed from HBM once per
 * token through y = W x products, as the paper frames the problem
 * (Kilictas & Alpay, "Bare-Metal Tensor Virtualization", arXiv 2601.03324,
 * §1 and §3.1). The weights live in one device arena filled by a single
 * host-to-device copy of a packed blob (§4.1, mmap'd model file; §3.2,
 * aligned buffers).
 *
 * Conventions for every entry point:
 *   - No exception crosses the ABI; every call returns a tvl_status.
 *     tvl_last_error() gives a message for the calling thread's last failure.
 *   - A tvl_model handle is not thread-safe: one host thread at a time.
 *   - "stream" arguments are cudaStream_t values passed as void*.
 *   - All tensors are float32; matrices are row-major [rows x cols].
 */
#ifndef TVL_H
#define TVL_H
#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  TVL_OK = 0,
  TVL_E_INVAL = 1,       /* bad argument or configuration */
  TVL_E_SIZE = 2,        /* blob size differs from tvl_blob_bytes() */
  TVL_E_ALIGN = 3,       /* pointer alignment the kernel needs is missing */
  TVL_E_NOMEM = 4,       /* device or pinned host allocation failed */
  TVL_E_CUDA = 5,        /* a CUDA runtime call failed (see tvl_last_error) */
  TVL_E_RANGE = 6,       /* token, position or step count out of range */
  TVL_E_TIMEOUT = 7,     /* a bounded device-side wait gave up; model unusable */
  TVL_E_UNSUPPORTED = 8  /* shape the GPU path does not handle (see tvl_load) */
} tvl_status;

/* Model shape. Paper §2.1: RMSNorm pre-normalisation, SwiGLU FFN with three
 * matrices, RoPE on q and k; §5.1: classifier tied to the token embedding. */
typedef struct {
  int32_t dim;          /* d, model width */
  int32_t hidden_dim;   /* F, SwiGLU hidden width */
  int32_t n_layers;     /* L (0 allowed: embedding -> final norm -> classifier) */
  int32_t n_heads;      /* H query heads; head_dim = d / H */
  int32_t n_kv_heads;   /* Hkv key/value heads; H % Hkv == 0 (query head h uses h / (H/Hkv)) */
  int32_t vocab_size;   /* V */
  int32_t max_seq;      /* S, KV-cache positions */
  double rope_theta;    /* RoPE base (10000) */
  double norm_eps;      /* RMSNorm epsilon, added to mean(x^2) inside the sqrt (1e-5, §11.2) */
  int32_t shared_classifier; /* 1 tied (Wcls is E), 0 untied, -1 infer from blob size (§5.1) */
  int32_t weight_bits;  /* 0: float32 weights as in the blob; 8: tvl_load turns every weight
                           matrix (and the embedding table) into 8-bit rows, as
                           tvl_quantize_q8 defines, and decodes with them; dim and
                           hidden_dim must then be multiples of 16; 4: the same with
                           4-bit rows as tvl_quantize_q4 defines (dim and hidden_dim
                           multiples of 32). Any other value is TVL_E_INVAL */
  int32_t max_batch;    /* sequences one launch may decode together, 0 or 1 (one) to 4;
                           each sequence slot gets its own KV cache and exchange buffers.
                           More than one needs weight_bits 0 */
} tvl_config;

typedef struct tvl_model tvl_model; /* opaque: device arena, stream, kernel plan */

/* Exact byte size of the packed blob for cfg, tied (1) or untied (0)
 * classifier; 0 if cfg is invalid.
 * Blob layout (the paper's "Tensor Virtualization Layout", §4.1, which it
 * leaves undefined; this is the definition used here): float32 row-major
 * tensors, each starting at a 128-byte-aligned offset (zero padding), in the
 * order  E[V x d];  per layer  g_att[d], Wq[d x d], Wk[kvd x d], Wv[kvd x d],
 * Wo[d x d], g_ffn[d], W1[F x d], W3[F x d], W2[d x F];  g_final[d];
 * Wcls[V x d] unless tied.  (kvd = Hkv * d / H.) */
size_t tvl_blob_bytes(const tvl_config* cfg, int32_t tied);

/* Load a model: pins `blob` (host memory owned by the caller, typically an
 * mmap of the model file, §4.1) if it is not pinned already, copies it with
 * ONE host-to-device transfer into a 256-byte-aligned device arena, builds
 * the RoPE table and zeroes the KV cache. On return the caller may free or
 * unmap `blob`.
 *   cfg        model shape; shared_classifier -1 takes the paper's heuristic
 *              (a blob one classifier short is tied).
 *   blob_bytes must equal tvl_blob_bytes(cfg, tied), else TVL_E_SIZE.
 *   stream     cudaStream_t for all work on this model; NULL: the library
 *              creates and owns a non-blocking stream.
 *   out        receives the handle (NULL on failure).
 * GPU-path requirements (else TVL_E_UNSUPPORTED): dim % 32 == 0,
 * head_dim % 4 == 0 and <= 128, hidden_dim % 4 == 0, max(dim, hidden_dim)
 * <= 16384. Invalid shapes give TVL_E_INVAL. Uses the current CUDA device. */
tvl_status tvl_load(const tvl_config* cfg, const void* blob, size_t blob_bytes, void* stream,
                    tvl_model** out);

/* Same, from a file: mmap(PROT_READ, MAP_PRIVATE | MAP_POPULATE) of `path`
 * (§4.1, and the Linux pre-fault hint of the artifact appendix), then
 * tvl_load on the mapping, then munmap. */
tvl_status tvl_load_file(const tvl_config* cfg, const char* path, void* stream, tvl_model** out);

/* One decode step (§7.1: the timed unit is one forward() call returning the
 * logits): embeds `token` at position `pos`, runs every layer (writing K/V
 * of this position into the cache) and the classifier.
 *   0 <= token < V and 0 <= pos < max_seq, else TVL_E_RANGE. Positions
 *   0..pos-1 must hold this sequence's K/V (call positions in order;
 *   calling a position again overwrites it).
 *   logits_out: V floats. Device pointer: the copy is queued on the model
 *   stream and the call returns without waiting. Host pointer: the call waits
 *   and then reports device-side errors; pinned, mapped, writable host
 *   memory (cudaHostAlloc, cudaHostRegister without the read-only flag) is
 *   written by the kernel itself, other host memory by a copy after it.
 *   NULL: logits stay on the device.
 * The whole step is one kernel launch (a persistent kernel). */
tvl_status tvl_forward(tvl_model* m, int32_t token, int32_t pos, float* logits_out);

/* Greedy decoding kept on the device (§9.1 names greedy decoding as the
 * baseline strategy; §7.1 generates 256 tokens): n_steps decode steps in ONE
 * kernel launch, starting with start_token at start_pos; the token fed at each
 * later step is the argmax of the previous logits (lowest index on ties).
 *   tokens_out: host array of n_steps; tokens_out[s] = argmax after step s.
 *   NULL: nothing is copied and the call does not wait.
 *   start_pos + n_steps <= max_seq, n_steps >= 1, else TVL_E_RANGE. */
tvl_status tvl_decode_greedy(tvl_model* m, int32_t start_token, int32_t start_pos,
                             int32_t n_steps, int32_t* tokens_out);

/* Batched decode: `batch` independent sequences (1 <= batch <= max_batch,
 * else TVL_E_INVAL) advance together, one position per step, in one kernel
 * launch that streams every weight once per step for all of them. The paper
 * (§ Implications for Computational Linguistics, "Enabling Advanced Decoding
 * Strategies") names beam search with B = 4 hypotheses as the case whose
 * bandwidth need grows B-fold when each hypothesis is decoded on its own;
 * here the B hypotheses share each step's single weight stream. Sequence b uses KV-cache slot b (slot 0
 * is the cache tvl_forward and tvl_decode_greedy use); all sequences are at
 * the same position pos and must have written positions 0..pos-1 of their
 * slots. Results per sequence equal a separate batch-1 run up to float
 * rounding (sums are taken in another order).
 * tvl_forward_batch: one step; tokens[b] (host array of batch) at position
 *   pos; logits_out [batch][V] (device pointer: queued, no wait; host: waits
 *   and reports device errors; NULL: kept on the device).
 * tvl_decode_greedy_batch: n_steps greedy steps from start_tokens[b] at
 *   start_pos; tokens_out (host, NULL allowed) [n_steps][batch]:
 *   tokens_out[s * batch + b] = argmax of sequence b's logits after step s.
 * Token out of range, pos < 0 or start_pos + n_steps > max_seq: TVL_E_RANGE. */
tvl_status tvl_forward_batch(tvl_model* m, int32_t batch, const int32_t* tokens, int32_t pos,
                             float* logits_out);
tvl_status tvl_decode_greedy_batch(tvl_model* m, int32_t batch, const int32_t* start_tokens,
                                   int32_t start_pos, int32_t n_steps, int32_t* tokens_out);

/* Multi-token prefill of sequence slot 0: tokens[0..n) (host array) at
 * positions start_pos .. start_pos + n - 1 run through every layer as one
 * block of n rows per layer, writing their K/V rows into the cache, and the
 * logits of the last position are returned — the same computation as n
 * tvl_forward calls (§2.1, §7.1), with each layer's weights read once for all
 * n positions. The products with the weight matrices run on the tensor
 * cores in float32 accuracy (as tvl_gemm: bf16 parts, fp32 accumulation);
 * the first call allocates the activations for max_seq positions (with the
 * partial sums of up to eight key ranges per query and head of the
 * attention, 4 * 8 * max_seq * H * (head_dim + 4) bytes) and the
 * bf16 parts of every layer's weight matrices (as many bytes as those
 * float32 matrices: 340 MB at 110M, 26 GB at 7B), kept until tvl_free; a
 * bounded wait that runs out in a product is reported by tvl_gemm_status.
 * Positions 0 .. start_pos - 1 must hold this sequence's K/V already.
 *   logits_out: V floats, as for tvl_forward (device: no wait; host: waits;
 *   NULL: kept on the device).
 *   n >= 1, start_pos >= 0, start_pos + n <= max_seq, tokens in [0, V), else
 *   TVL_E_RANGE; a model loaded with weight_bits 8 or 4: TVL_E_UNSUPPORTED. */
tvl_status tvl_prefill(tvl_model* m, const int32_t* tokens, int32_t n, int32_t start_pos,
                       float* logits_out);

/* Standalone GEMV y = W x (§6.1), W [d_out x d_in] row-major, x [d_in],
 * y [d_out]; all device pointers; queued on `stream` (NULL = default stream),
 * does not wait. d_out >= 1, d_in >= 1, else TVL_E_INVAL. The fast path
 * (TMA bulk staging) needs W and x 16-byte aligned and d_in % 4 == 0 and
 * d_in <= 16384; other shapes take a plain per-row kernel. Deterministic: the
 * same inputs give the same bits. A per-stream scratch buffer (a few KB) is
 * allocated on first use for matrices with fewer rows than the GPU has SMs
 * (split along d_in) and kept until exit; concurrent calls on different
 * streams are safe. The kernel is launched with a programmatic dependency on
 * the stream's previous kernel: it may start while that kernel finishes, and
 * reads x, writes y and copies W only once that kernel has completed. */
tvl_status tvl_gemv(const float* W, const float* x, float* y, int32_t d_out, int32_t d_in,
                    void* stream);

/* Y = X W^T for a block of n vectors (the products of a multi-token prefill,
 * §2.1 and §7.1: n decode steps whose weight reads are shared), on the
 * tensor cores (tcgen05) in float32 accuracy: each float is split into two
 * bf16 parts (hi = bf16(a), lo = bf16(a - hi)) and the three products
 * hi*hi + hi*lo + lo*hi are accumulated in fp32; what is dropped is about
 * 2^-16 of each product. W [M x K], X [n x K], Y [n x M], row-major float32,
 * device pointers, 16-byte aligned; K % 8 == 0 (else TVL_E_UNSUPPORTED);
 * n, M, K >= 1 (else TVL_E_INVAL). Queued on `stream`, does not wait. A
 * per-stream scratch buffer for the bf16 parts (4 (M + n) K bytes) is
 * allocated on first use and grown when needed, kept until exit. */
tvl_status tvl_gemm(const float* W, const float* X, float* Y, int32_t n, int32_t M, int32_t K,
                    void* stream);

/* Waits for `stream`, then reports (and clears) the tensor-core GEMM's error
 * word: TVL_E_TIMEOUT if a bounded wait inside a tvl_gemm or prefill product
 * ran out since the last query (that call's Y is incomplete), else TVL_OK. */
tvl_status tvl_gemm_status(void* stream);

/* Weight-only 8-bit rows (also the weight format of a model loaded with
 * weight_bits = 8). The paper leaves quantization to future work
 * (§ Future Work: Quantization: narrow weights unpacked on the fly, for less
 * memory traffic per token); this is one reading of it. A matrix W [rows x
 * cols] becomes packed rows of 16 + cols bytes each: the float32 scale
 * s = max_j |W[r][j]| / 127 (bytes 0-3), twelve zero bytes, then the codes
 * q[r][j] = the integer nearest to W[r][j] / s (ties to even, in [-127, 127];
 * an all-zero row has s = 0 and codes 0), every step in float32. The code
 * stands for the weight s * q. cols must be a positive multiple of 16.
 * tvl_q8_bytes: bytes of the packed rows (0 if rows < 1 or cols is invalid). */
size_t tvl_q8_bytes(int32_t rows, int32_t cols);

/* Quantize W (device, float32, row-major, 16-byte aligned) into Wq8 (device,
 * tvl_q8_bytes(rows, cols) bytes, 16-byte aligned), on `stream`, without
 * waiting. Errors: TVL_E_INVAL (null pointer, bad size), TVL_E_ALIGN. */
tvl_status tvl_quantize_q8(const float* W, void* Wq8, int32_t rows, int32_t cols, void* stream);

/* y = W' x for the weights W' the packed rows stand for (y[r] = s_r * sum_j
 * q[r][j] x[j]); Wq8 and x device pointers, 16-byte aligned; d_in a multiple
 * of 16 and at most 16368 (a packed row fits one 16 KB stage), else
 * TVL_E_INVAL / TVL_E_UNSUPPORTED. Queued on `stream`, does not wait,
 * allocates nothing. */
tvl_status tvl_gemv_q8(const void* Wq8, const float* x, float* y, int32_t d_out, int32_t d_in,
                       void* stream);

/* Weight-only 4-bit rows: the same reading of the paper's quantization
 * future work (§ Future Work: Quantization names 4-bit weights unpacked on
 * the fly) with 7 levels on each side of zero. A matrix W [rows x cols]
 * becomes packed rows of 16 + cols/2 bytes: the float32 scale
 * s = max_j |W[r][j]| / 7 (bytes 0-3), twelve zero bytes, then the codes
 * q[r][j] = the integer nearest to W[r][j] / s (ties to even, in [-7, 7]; an
 * all-zero row has s = 0 and codes 0), every step in float32, two per byte as
 * 4-bit two's complement: byte m holds column 2m in its low nibble and column
 * 2m + 1 in its high nibble. The code stands for the weight s * q. cols must
 * be a positive multiple of 32. tvl_q4_bytes: bytes of the packed rows (0 if
 * rows < 1 or cols is invalid). */
size_t tvl_q4_bytes(int32_t rows, int32_t cols);

/* Quantize W (device, float32, row-major, 16-byte aligned) into Wq4 (device,
 * tvl_q4_bytes(rows, cols) bytes, 16-byte aligned), on `stream`, without
 * waiting. Errors: TVL_E_INVAL (null pointer, bad size), TVL_E_ALIGN. */
tvl_status tvl_quantize_q4(const float* W, void* Wq4, int32_t rows, int32_t cols, void* stream);

/* y = W' x for the weights W' the packed 4-bit rows stand for (y[r] = s_r *
 * sum_j q[r][j] x[j]); Wq4 and x device pointers, 16-byte aligned; d_in a
 * multiple of 32 and at most 32736 (a packed row fits one 16 KB stage), else
 * TVL_E_INVAL / TVL_E_ALIGN / TVL_E_UNSUPPORTED. Queued on `stream`, does not
 * wait, allocates nothing. */
tvl_status tvl_gemv_q4(const void* Wq4, const float* x, float* y, int32_t d_out, int32_t d_in,
                       void* stream);

/* tvl_gemv without any allocation. The paper has no counterpart: this entry
 * exists for callers that cannot allocate device memory at call time — a host
 * thread that must not stall other streams (cudaMalloc and cudaFree may
 * synchronise the device implicitly), or a caller that has handed all device
 * memory to its own pool (tvl_gemv's first short-and-wide call on a stream
 * allocates its scratch and could fail there).
 * Same arguments, layout, paths and results as tvl_gemv (same kernel, same
 * split, bit-identical output). The split-K scratch is one static module
 * array of 48 KB per device (8192 partials, 4096 row counters), not
 * allocated memory. A shape whose split needs more (never on a 152-SM GB300:
 * at most 302 partials and 151 rows) returns TVL_E_UNSUPPORTED with the
 * sizes in tvl_last_error(); use tvl_gemv for it.
 * The FIRST call on a device does a one-time setup: it looks up the array's
 * device address, zeroes its counters on `stream` and waits for that, so make
 * it before any work that must not wait (e.g. before a stream capture).
 * The scratch is shared by every call on the device: calls that can overlap
 * on the device (different streams without ordering between them) race on it
 * and give wrong results; order them, or use tvl_gemv. */
tvl_status tvl_gemv_noalloc(const float* W, const float* x, float* y, int32_t d_out,
                            int32_t d_in, void* stream);

/* Error report of the standalone GEMV calls (tvl_gemv, tvl_gemv_noalloc,
 * tvl_gemv_q8, tvl_gemv_q4), which queue their kernel and return without
 * waiting. Every wait inside those kernels is bounded (one second); when one
 * runs out — only a broken device can cause it — the kernel raises
 * TVL_E_TIMEOUT in an error word of the current device and its CTAs leave, so
 * that call's y is incomplete. This call waits for the work queued on
 * `stream`, then returns that error (and clears it) or TVL_OK. Split-K
 * counters are tagged with their call, so calls after a failed one are
 * correct whether or not this is called. Allocates nothing. */
tvl_status tvl_gemv_status(void* stream);

/* Failure-detection self-test of the standalone GEMV kernel: tvl_gemv_noalloc's
 * kernel (same shape rules, same static scratch) runs with the last stage of
 * CTA 0 never copied, so that CTA's consumer waits for it until the one-second
 * limit runs out. Returns what tvl_gemv_status then reports: TVL_E_TIMEOUT
 * expected, with the CUDA context still usable; y is left partly written.
 * W, x, y as for tvl_gemv (a shape the streaming kernel takes, else
 * TVL_E_UNSUPPORTED). */
tvl_status tvl_selftest_gemv_timeout(const float* W, const float* x, float* y, int32_t d_out,
                                     int32_t d_in, void* stream);

/* Wait for the model's queued work, then report any device-side error. */
tvl_status tvl_sync(tvl_model* m);

/* Release the device arena and the stream the library created. NULL is ignored. */
void tvl_free(tvl_model* m);

const char* tvl_status_string(tvl_status s);
const char* tvl_last_error(void);

/* Facts about a loaded model, for benchmarks and tests. */
typedef struct {
  int64_t arena_bytes;       /* the single device allocation */
  int64_t weight_bytes;      /* the blob as copied */
  int64_t streamed_bytes;    /* weight bytes read per decode step */
  int32_t grid;              /* persistent CTAs (one per SM) */
  int32_t threads;           /* threads per CTA */
  int32_t smem_bytes;        /* dynamic shared memory per CTA */
  int32_t ring_stages;       /* weight staging ring: stages x stage_bytes */
  int32_t stage_bytes;
  int32_t tied;
  int32_t exchanges_per_step; /* tagged exchanges between CTAs in one greedy step */
  int32_t max_batch;          /* as loaded (1 when the config said 0) */
  int64_t next_tag;           /* exchange tag the next launch starts from (1 .. 2^32 - 1) */
} tvl_model_info;
tvl_status tvl_get_info(const tvl_model* m, tvl_model_info* out);

/* Device timestamps (ns, %globaltimer) taken at the end of each step of the
 * last tvl_decode_greedy call, for per-step latency statistics (§7.3). */
tvl_status tvl_step_times(tvl_model* m, uint64_t* ns_out, int32_t n);

/* Failure-detection self-test: the decode kernel's bounded exchange poll
 * (the consumer warps of one CTA polling a tagged word) waits on a word that
 * nothing writes, with a wait limit of limit_ms (1 .. 10000). Expected result
 * TVL_E_TIMEOUT, raised by the kernel itself, with the CUDA context still
 * usable. Uses the current device. */
tvl_status tvl_selftest_barrier_timeout(int32_t limit_ms);

/* ---- Test hooks: not needed for normal use ---------------------------------
 * They reach states that are otherwise hours of decoding or an out-of-memory
 * device away. The paper has no counterpart. */

/* Makes the k-th device or pinned-host allocation attempt of the library from
 * now on fail as if memory were exhausted (k = 0: the next attempt); k < 0
 * disarms. It fires once. Lets a test reach every failure point of tvl_load,
 * tvl_prefill and tvl_gemv, which must then return TVL_E_NOMEM and hold no
 * allocation. Process-wide; not thread-safe against concurrent loads. */
void tvl_debug_fail_allocation(int32_t k);

/* Device and pinned-host allocations the library holds right now (arenas,
 * prefill activations, GEMV scratch buffers). */
int64_t tvl_debug_live_allocations(void);

/* Sets the exchange tag the model's next launch starts from (tvl_model_info.
 * next_tag), 1 .. 2^32 - 1, else TVL_E_INVAL. Tags are 32-bit and 0 marks a
 * word never written: a launch whose tags would pass 2^32 - 1 first zeroes
 * the exchange words on the model's stream and starts again from tag 1. This
 * hook puts a model next to that point without 2^32 exchanges of decoding.
 * A tag below the model's next one also zeroes the exchange words first
 * (queued on the model's stream), since published words only grow. */
tvl_status tvl_debug_set_next_tag(tvl_model* m, uint64_t tag);

#ifdef __cplusplus
}
#endif
#endif /* TVL_H */

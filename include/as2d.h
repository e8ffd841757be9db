/*
 * as2d.h -- C-ABI of the GB300 (sm_103a) target-side block verification
 * library, libas2d.so.
 *
 * The operation (paper: Section 3.2 "Target verification"; App. A.2
 * "Configuration and execution boundaries"; App. C.2 "Verification and state
 * repair"; App. C.4, Eq. 3 and Prop. 1):
 *   the target decoder holds a committed prefix in its KV cache (prefilled
 *   audio and instruction tokens plus every committed token except the last
 *   one) and a pending "known root" token -- the last committed token, not yet
 *   forwarded.  A verification call forwards the root followed by k drafter
 *   candidates c_1..c_k in one causal pass (physical width K = k + 1),
 *   takes the greedy token g_i after each row i, accepts the longest prefix
 *   c_1..c_n with c_{i+1} = g_i, and emits the correction g_n (the bonus
 *   token when n = k).  The cache keeps the root's and the accepted
 *   candidates' entries; the rejected rows' entries are dropped.  The
 *   correction is not forwarded: it becomes the next call's root, so full
 *   acceptance needs no extra single-token call (App. C.2, known-root
 *   carry).  With k = 0 the call is one plain greedy decode
 *   step of Eq. 3.
 *
 * Conventions shared by every entry point:
 *   - Pointers documented "device" are CUDA device pointers on the current
 *     device; "host" pointers are ordinary host memory, read before the call
 *     returns.  `stream` is a cudaStream_t (NULL = the legacy default stream).
 *   - Work is enqueued on `stream` and never synchronises with the host,
 *     except where an entry point says it does.  Device outputs are valid once
 *     the caller synchronises the stream.
 *   - Argument errors are found on the host before anything is enqueued and
 *     leave all state unchanged.  as2d_last_error() then describes the error
 *     (thread-local).
 *   - Every bf16 value is the upper 16 bits of an IEEE float (bfloat16).
 */
#ifndef AS2D_H
#define AS2D_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t as2d_status;
#define AS2D_OK 0
#define AS2D_ERR_INVALID_ARG (-1)   /* bad pointer, size or value            */
#define AS2D_ERR_CAPACITY (-2)      /* L + k + 1 would exceed the capacity   */
#define AS2D_ERR_CUDA (-3)          /* a CUDA runtime call failed            */
#define AS2D_ERR_UNSUPPORTED (-4)   /* shape outside what the kernels handle */
#define AS2D_ERR_DEVICE (-5)        /* a kernel reported an error or timeout */
#define AS2D_ERR_NO_MEMORY (-6)     /* a host allocation failed              */

/* Device-side error bits (as2d_kv_check's message names them; the static
   decode step returns them through its error_bits output). */
#define AS2D_DEVERR_BAD_TOKEN 1  /* a root or candidate id outside [0, vocab)  */
#define AS2D_DEVERR_ROLLBACK 2   /* a rollback beyond the committed length     */
#define AS2D_DEVERR_TIMEOUT 4    /* a kernel's bounded wait gave up            */
#define AS2D_DEVERR_CAPACITY 8   /* a device-side length left no room for the
                                    call's rows (length < 0 or length + rows >
                                    capacity): that request was skipped       */

/* Largest number of candidates per request in one call (the budget b of
   App. A.2; physical width K = k + 1 <= 17). */
#define AS2D_MAX_K 16
/* Largest number of requests verified together in one call. */
#define AS2D_MAX_BATCH 64

/* Decoder shape.  Requirements: hidden % 128 == 0, (n_q * head_dim) % 128
   == 0, ffn % 64 == 0, vocab % 8 == 0, head_dim in {64, 128},
   n_q % n_kv == 0, n_kv * head_dim % 128 == 0.  rope_theta is the rotary base (rotate-half
   pairing of dimensions i and i + head_dim/2, angle pos * theta^(-2i/d));
   rms_eps is added to the mean square before the root. */
typedef struct as2d_config {
  int32_t n_layers, hidden, n_q_heads, n_kv_heads, head_dim, ffn, vocab;
  float rope_theta, rms_eps;
} as2d_config;

/* Weights, as device pointers to bf16 in checkpoint (logical) layouts,
   row-major: embed, lm_head [vocab][hidden]; final_norm and the per-layer
   attn_norm, mlp_norm gains [hidden]; w_q [n_q*d][hidden], w_k, w_v
   [n_kv*d][hidden] (head j in rows [j*d, (j+1)*d)); w_o [hidden][n_q*d];
   w_gate, w_up [ffn][hidden]; w_down [hidden][ffn].  The per-layer members
   are HOST arrays of n_layers device pointers.  as2d_model_load copies every
   tensor into memory the model owns (re-laid out for the kernels); the caller
   may free its buffers once as2d_model_load has returned. */
typedef struct as2d_weights {
  const void* embed;
  const void* final_norm;
  const void* lm_head;
  const void* const* attn_norm;
  const void* const* w_q;
  const void* const* w_k;
  const void* const* w_v;
  const void* const* w_o;
  const void* const* mlp_norm;
  const void* const* w_gate;
  const void* const* w_up;
  const void* const* w_down;
} as2d_weights;

typedef struct as2d_model as2d_model;
typedef struct as2d_kv as2d_kv;

/* Outputs of one verification call.  rows = sum over requests of (k_b + 1),
   ordered request by request, each request's root row first.
   n_accepted, correction_token: device int32 [batch] (required).
   greedy: device int32 [rows], the greedy token after each row (nullable).
   logits: device float [rows][vocab], fp32 logits of every row (nullable;
   the paper's full-logits verification of App. B.2 stores [1, K, vocab]). */
typedef struct as2d_verify_out {
  int32_t* n_accepted;
  int32_t* correction_token;
  int32_t* greedy;
  float* logits;
} as2d_verify_out;

/* Load a model onto the current device.  Synchronises the device before it
   returns.  On success *out owns its device memory until as2d_model_free. */
as2d_status as2d_model_load(const as2d_config* cfg, const as2d_weights* w,
                            as2d_model** out);

/* Size this model's kernel grids for n_sms SMs (1 .. the device's count; the
   default is the device's count), so that the pass can share the GPU with
   other work confined to the remaining SMs -- for example a drafter on its
   own stream (as2d_session_run).  The work split depends on (shape, n_sms)
   only: results stay batch invariant and bit-identical for a given budget;
   another budget adds partial sums in another order.  States created before
   a larger budget was set refuse to run (AS2D_ERR_INVALID_ARG): set the
   budget before as2d_kv_init_prefilled. */
as2d_status as2d_model_set_sm_budget(as2d_model* model, int32_t n_sms);

/* Bind a verification state of `batch` requests to a caller-allocated cache
   and its prefilled prefix (App. A.1: the retained audio KV plus the
   instruction, a valid prefix of the reference prompt).
   k_cache, v_cache: device bf16, layout [n_layers][batch][n_kv][capacity]
   [head_dim]; positions [0, kv_len[b]) of request b hold its prefilled keys
   (already rotated to their positions) and values.  The library writes the
   entries of forwarded rows; the caller keeps both buffers alive until
   as2d_kv_free.  kv_len, root_tokens: host int32 [batch]; root_tokens[b] is
   request b's pending known root (the first token chosen after prefill).
   capacity <= 65536 (AS2D_ERR_UNSUPPORTED above).  Allocates the state's
   device working memory.  Synchronises the device. */
as2d_status as2d_kv_init_prefilled(as2d_model* model, int32_t batch,
                                   const int32_t* kv_len, int32_t capacity,
                                   void* k_cache, void* v_cache,
                                   const int32_t* root_tokens, as2d_kv** out);

/* Verify one block per request (Section 3.2; App. C.2).
   candidates: device int32, packed: request b's k_b candidates start at
   index sum_{b' < b} k_{b'}.  k: host int32 [batch], 0 <= k_b <= AS2D_MAX_K.
   Request b forwards rows [root_b, c_1..c_{k_b}] at positions
   L_b .. L_b + k_b and afterwards holds L_b' = L_b + n_b + 1 and
   root_b' = correction_b, all on the device.  The host keeps only an upper
   bound of L_b (it grows by k_b + 1 per call); AS2D_ERR_CAPACITY is returned
   when that bound plus k_b + 1 would exceed the capacity (as2d_kv_read_state
   refreshes the bound).  Candidate ids outside [0, vocab) are a device-side
   error (as2d_kv_check).  Results are batch invariant: each row's logits are
   bitwise the same whatever the other rows of the call. */
as2d_status as2d_verify_block(as2d_kv* kv, const int32_t* candidates,
                              const int32_t* k, const as2d_verify_out* out,
                              void* stream);

/* Instruction-suffix prefill (App. A.1: processing the instruction with the
   retained, compatible audio KV gives the initial decoding state): forwards
   tokens[0..n) (device int32 [n], ids in [0, vocab)) at positions
   L .. L + n - 1 of a batch-1 state and keeps every entry, in passes of up
   to 64 rows through the verification pass (the first call allocates a
   working state for such passes, kept until as2d_kv_free; its attention
   buffers grow with the capacity, about 0.9 MB per 64 positions for the
   7B shape).  The pending root
   before the call is discarded; afterwards L' = L + n and the root is the
   greedy token after tokens[n - 1] -- the first token of the response --
   also written to first_token (device int32 [1]) unless it is NULL.
   AS2D_ERR_UNSUPPORTED for batch > 1, AS2D_ERR_CAPACITY when the length
   bound plus n exceeds the capacity; bad token ids are device errors
   (as2d_kv_check).  Asynchronous on `stream`. */
as2d_status as2d_prefill(as2d_kv* kv, const int32_t* tokens, int32_t n,
                         int32_t* first_token, void* stream);

/* One greedy decode step for every request: as2d_verify_block with all
   k_b = 0 (App. C.2: with no ready candidate the target advances alone by one
   token). */
as2d_status as2d_decode_step(as2d_kv* kv, const as2d_verify_out* out,
                             void* stream);

/* Restore each request's state to an earlier committed prefix (App. C.4,
   requirement 2): length new_len[b] and pending root new_root[b] (host int32
   [batch]).  Entries [0, new_len[b]) must be ones this state holds; a
   new_len above the device-side length is a device error that leaves that
   request unchanged.  Asynchronous on `stream`. */
as2d_status as2d_kv_rollback(as2d_kv* kv, const int32_t* new_len,
                             const int32_t* new_root, void* stream);

/* Synchronise `stream`, copy the device-side lengths and roots into host
   int32 [batch] arrays (either may be NULL) and reset the host's length
   bounds to them. */
as2d_status as2d_kv_read_state(as2d_kv* kv, int32_t* len, int32_t* root,
                               void* stream);

/* Device pointers to the state's int32 [batch] lengths and roots, for
   consumers on the device (e.g. a drafter kernel that builds the next block
   without a host round trip).  Read-only for the caller. */
as2d_status as2d_kv_device_state(as2d_kv* kv, const int32_t** len,
                                 const int32_t** root);

/* Synchronise `stream` and return AS2D_ERR_DEVICE if any kernel of this
   state reported an error since the last check (then cleared), else
   AS2D_OK. */
as2d_status as2d_kv_check(as2d_kv* kv, void* stream);

/* Time limit, in nanoseconds, of the waits inside the kernels of this state's
   calls for a bulk copy, a tensor-core product or an accumulator (default
   2 s; this file's failure detection, not a paper mechanism).  A wait that
   runs out records AS2D_DEVERR_TIMEOUT, reported by as2d_kv_check, and its
   block of threads abandons that call's work: the call's outputs are then
   undefined, and the state should be restored with as2d_kv_rollback.  The
   waits by which a block drains its own outstanding copies and products
   before it ends keep the 2 s limit, so none is outstanding when it exits.
   A limit of 0 makes every wait that is not already satisfied give up at
   once, which exercises the failure path.  Takes effect for later calls. */
as2d_status as2d_kv_set_wait_limit(as2d_kv* kv, uint64_t ns);

/* One greedy decode step (k = 0) of a single request that allocates no
   memory.  The paper has no counterpart: this is for callers that must not
   allocate device memory when they decode -- for example a process whose
   device memory is handed out by another component under a fixed budget, or
   a real-time loop that cannot accept the latency or the possible failure of
   an allocation.  The model must have been loaded (as2d_model_load allocates,
   once, at set-up).  Every other byte a call needs lives in one array of
   9,735,424 bytes compiled into the library; each GPU that loads the library
   holds it until the process exits.
   k_cache, v_cache: device bf16 [n_layers][1][n_kv][capacity][head_dim] as
   for as2d_kv_init_prefilled.  len, root: device int32 [1], the request's
   state, updated in place (len += 1, root = correction) as by
   as2d_decode_step; *len must lie in [0, capacity - 1] when the step runs.
   correction_token: device int32 [1].  logits: device float [vocab] or NULL.
   error_bits: device int32 [1] or NULL; receives the step's AS2D_DEVERR_*
   bits (0 when it ran cleanly).
   Limits (AS2D_ERR_CAPACITY / AS2D_ERR_UNSUPPORTED on the host, before any
   work): capacity <= 4096, hidden <= 4096, ffn <= 20480, n_q * head_dim <=
   4096, n_kv <= 8, n_q / n_kv <= 16, vocab <= 262144, at most 192 SMs.
   The length lives on the device, so the host cannot check it: the kernels
   do.  A step whose *len is outside [0, capacity - 1], or whose root is
   outside [0, vocab), writes nothing to the cache, leaves len and root as
   they were, sets *correction_token to -1 and reports AS2D_DEVERR_CAPACITY
   (or AS2D_DEVERR_BAD_TOKEN) in error_bits.
   The first call on a device (and the first after a model of another shape)
   looks up the array's device address and builds descriptors of it; make
   that first call before any stream capture.  Calls from several host
   threads are enqueued one at a time, but all calls share the one array and
   each starts by clearing the parts that must start at zero, so calls that
   overlap on the GPU (other streams) race and give wrong results: issue
   them one after another on one stream, or synchronise between them.
   Device-side errors of this entry point are reported only through
   error_bits, not through as2d_kv_check. */
as2d_status as2d_decode_step_static(as2d_model* model, void* k_cache, void* v_cache,
                                    int32_t capacity, int32_t* len, int32_t* root,
                                    int32_t* correction_token, float* logits,
                                    int32_t* error_bits, void* stream);

/* Measurement support (not part of the verification step).  Kernel classes
   of one verification pass, in launch order per layer: */
#define AS2D_KERNEL_QKV 0        /* norm + QKV projection               */
#define AS2D_KERNEL_ATTENTION 1  /* RoPE + KV append + attention        */
#define AS2D_KERNEL_O 2          /* output projection + residual        */
#define AS2D_KERNEL_GATE_UP 3    /* norm + gate/up projection + SwiGLU   */
#define AS2D_KERNEL_DOWN 4       /* down projection + residual          */
#define AS2D_KERNEL_LM_HEAD 5    /* final norm + LM head + argmax       */
#define AS2D_KERNEL_OTHER 6      /* embedding gather, accept scan, ...  */
#define AS2D_KERNEL_CLASSES 7

/* Record a CUDA event pair on the call's stream around the launches of
   kernel class `kernel_class` (one pair per layer, or per call for the LM
   head) in later calls (-1 stops recording).  Also
   counts every kernel the library launches.  Events are created on demand. */
as2d_status as2d_kv_profile(as2d_kv* kv, int32_t kernel_class);

/* Synchronise the recorded events and return the number of recorded
   event pairs of the class, their summed device time in milliseconds, and the
   number of kernels the library launched since the last read; then reset. */
as2d_status as2d_kv_profile_read(as2d_kv* kv, int32_t* launches,
                                 double* total_ms, int64_t* all_launches);

void as2d_kv_free(as2d_kv* kv);
void as2d_model_free(as2d_model* model);

/* ---- Candidate buffer, read cursor and alignment -------------------------
   (Section 3.1 "Ordered publication and buffering"; Section 3.2 "Candidate
   alignment"; App. C.1 "Source records and incremental publication"; App. C.3
   "Candidate alignment"; Fig. 4.)  Host-side: one buffer per request and
   source.  The producer appends immutable batches of at most
   AS2D_CBUF_BATCH tokens; verification reads a snapshot of what is published
   from a read cursor that only alignment moves.  Alignment changes the
   cursor, never published tokens, committed tokens or the target's state, so
   the committed text is the target's greedy text whatever the buffer holds
   (Prop. 1).  Every entry point below is safe to call from several host
   threads at once (a producer thread publishing while the verifier reads):
   each one is atomic with respect to the others on the same buffer.

   Alignment, after a call that verified k candidates from cursor c,
   accepted n of them and ended with the target's token x (the correction,
   or the bonus token when n == k), with search bound W (the window):
     R1  x stands at buffer position m = c + n.  Once the buffer holds x at m
         (possible only after full acceptance; re-checked at each
         as2d_cbuf_candidates until m is published), the cursor steps over it
         to m + 1.
     R2  Otherwise m stays eligible: the next call verifies root x followed by
         the candidates from m (x may be a target insertion); if it accepts
         n >= 1, R1 applies to it.
     R3  If it accepts none, its token t is the first alignment anchor: the
         cursor moves to j + 1 for the first j in (m, m + W] holding t, else
         to j + 2 for the first j in [m, m + W] holding x, else the target
         decodes alone (k = 0).  While it does, its latest token is looked for
         before each call in the published positions [s, s + W) upwards, then
         [max(f, s - W), s) downwards, where f = m + 1 is where it began
         decoding alone and s starts at f and grows by one per token decoded
         alone; a match at j moves the cursor to j + 1. */
#define AS2D_CBUF_BATCH 8
#define AS2D_CBUF_NORMAL 0   /* candidates follow the cursor              */
#define AS2D_CBUF_REALIGN 1  /* R1/R2: waiting on the token at m          */
#define AS2D_CBUF_ALONE 2    /* R3: no usable candidates; k = 0           */

/* Source record of one published batch (App. C.1).  confidence is
   meaningful only when has_confidence != 0. */
typedef struct as2d_source_record {
  int32_t request, source, producer, offset;
  double time;
  float confidence;
  int32_t has_confidence;
} as2d_source_record;

typedef struct as2d_cbuf as2d_cbuf;

/* Create an empty buffer with search bound `window` in [1, 1024]. */
as2d_status as2d_cbuf_create(int32_t window, as2d_cbuf** out);

/* Append one batch: tokens host int32 [n], 1 <= n <= AS2D_CBUF_BATCH, every
   id >= 0; rec (host, required) is copied.  Published tokens never change. */
as2d_status as2d_cbuf_publish(as2d_cbuf* buf, const int32_t* tokens, int32_t n,
                              const as2d_source_record* rec);

/* The candidates for the next verification call: applies the checks that
   wait on publication (R1's step-over, R3's search while decoding alone),
   then copies up to b (0 <= b <= AS2D_MAX_K) published tokens from the cursor
   into host int32 tokens[b] and their number into *k (0 while the target
   decodes alone).  The next as2d_cbuf_after_call must report that k. */
as2d_status as2d_cbuf_candidates(as2d_cbuf* buf, int32_t b, int32_t* tokens,
                                 int32_t* k);

/* Report the call's outcome: the k of the last as2d_cbuf_candidates,
   n_accepted in [0, k] and the call's final token (correction or bonus,
   >= 0).  Moves the cursor by R1-R3. */
as2d_status as2d_cbuf_after_call(as2d_cbuf* buf, int32_t k, int32_t n_accepted,
                                 int32_t correction);

/* Published token count, cursor and mode (AS2D_CBUF_*); any may be NULL. */
as2d_status as2d_cbuf_state(as2d_cbuf* buf, int32_t* ready, int32_t* cursor,
                            int32_t* mode);

/* Tokens and batch records the buffer still holds (either may be NULL).
   Positions stay absolute, but tokens below both the cursor and the
   alignment position -- which no rule reads again -- are dropped once 4096
   of them have gathered, with the records of the batches wholly below them
   (App. C.1: exhausted records are discarded; the others keep their order
   and provenance), so a long session holds a bounded buffer. */
as2d_status as2d_cbuf_held(as2d_cbuf* buf, int32_t* tokens, int32_t* records);

/* Copy the source record of the batch that published `position`
   (AS2D_ERR_INVALID_ARG if the position is not published or was dropped). */
as2d_status as2d_cbuf_source_of(as2d_cbuf* buf, int32_t position,
                                as2d_source_record* out);

void as2d_cbuf_free(as2d_cbuf* buf);

/* One verification call driven by candidate buffers: bufs is a host array of
   kv's batch buffers (request r reads bufs[r]).  Takes up to b candidates
   from each buffer, copies them to the device, runs as2d_verify_block on
   `stream`, reads n_accepted and the correction back (this synchronises the
   stream) and reports them to each buffer.  Outputs (host, may be NULL):
   k_used int32 [batch]; committed int32 [batch][b + 1], row r holding the
   request's n_r + 1 committed tokens (accepted candidates, then the
   correction); n_committed int32 [batch] = n_r + 1.  The host's length
   bounds are tightened with the read-back n_r.  Device staging memory
   is allocated on the first call and kept until as2d_kv_free.  Errors of
   as2d_verify_block are returned as they are, before any buffer changes. */
as2d_status as2d_verify_from_buffers(as2d_kv* kv, as2d_cbuf* const* bufs, int32_t b,
                                     int32_t* k_used, int32_t* committed,
                                     int32_t* n_committed, void* stream);

/* ---- Producer / verifier sessions and their time accounting --------------
   (App. D.2 "Overlap, added work, and performance limits": the service
   intervals, D, V, O, H and the identity T = D + V - O + H;
   Section 3.1: the producer runs without target feedback and the target
   never waits for it.) */

/* A small decoder on the host cores: a producer placed on a different
   processor than the target, as the paper places drafter and target on
   different processors of one device.  fp32, one greedy decode step per
   call over its own cache (positions 0, 1, ...), matrix-vector products
   split over `threads` OpenMP threads.  w holds HOST float arrays in the
   layouts of as2d_weights (per-layer members: host arrays of host pointers);
   they are copied.  The shape rules of as2d_config do not apply (any
   positive sizes, n_q % n_kv == 0, even head_dim). */
typedef struct as2d_cpu_decoder as2d_cpu_decoder;
as2d_status as2d_cpu_decoder_create(const as2d_config* cfg, const as2d_weights* w,
                                    int32_t capacity, int32_t threads, int32_t root,
                                    as2d_cpu_decoder** out);
/* Forward the pending root at the next position, append its keys and values,
   make the greedy token the new root and return it in *token_out (may be
   NULL).  AS2D_ERR_CAPACITY when the cache is full. */
as2d_status as2d_cpu_decoder_step(as2d_cpu_decoder* d, int32_t* token_out);
/* The last step's logits: host float [vocab]. */
as2d_status as2d_cpu_decoder_logits(as2d_cpu_decoder* d, float* logits);
/* Back to an earlier length (<= the current one) with pending root `root`. */
as2d_status as2d_cpu_decoder_reset(as2d_cpu_decoder* d, int32_t len, int32_t root);
void as2d_cpu_decoder_free(as2d_cpu_decoder* d);

/* Service-interval accounting over [0, T].  p: host double [np][2] producer
   service intervals (start, end); v: host double [nv][2] verifier
   intervals; each is clipped to [0, T] and merged with the overlapping
   intervals of its own set.  out: host double [5] receives D = |P|, V = |V|,
   O = |P n V|, H = |[0, T] \ (P u V)| and T, so that T = D + V - O + H.
   AS2D_ERR_INVALID_ARG for an interval with end < start, T < 0 or counts
   < 0. */
as2d_status as2d_interval_accounting(const double* p, int32_t np, const double* v,
                                     int32_t nv, double T, double* out);

/* One request decoded to n_commit tokens by a producer publishing into a
   candidate buffer and a verifier drawing from it. */
typedef struct as2d_session_spec {
  as2d_kv* target;        /* batch-1 target state, advanced by the session          */
  as2d_kv* drafter;       /* batch-1 drafter state, one k = 0 decode step per
                             produced token on drafter_stream; NULL = no drafter
                             compute (tokens are published as fast as scripted)  */
  as2d_cbuf* buf;         /* the request's candidate buffer, written by the session */
  const int32_t* script;  /* host [n_script]: the token published by producer step i */
  int32_t n_script;
  int32_t b;              /* candidates per verification call, 0..AS2D_MAX_K       */
  int32_t publish_every;  /* producer steps per published batch, 1..AS2D_CBUF_BATCH */
  int32_t n_commit;       /* stop once at least this many tokens are committed     */
  int32_t overlapped;     /* 1: the producer runs on its own host thread and stream
                             alongside the verifier; 0: serial comparator -- the
                             producer runs (one batch) only while the verifier
                             waits, whenever fewer than b candidates are ready    */
  void* target_stream;
  void* drafter_stream;
  as2d_cpu_decoder* cpu_drafter;  /* when not NULL (and drafter is NULL): one
                                     host-core decode step per produced token */
} as2d_session_spec;

typedef struct as2d_session_stats {
  double T, D, V, O, H;   /* seconds: the accounting above over the session     */
  int32_t rounds;         /* verification calls (target-only rounds included)   */
  int32_t alone_rounds;   /* calls with k = 0                                    */
  int32_t committed;      /* tokens committed (accepted + one per call)          */
  int32_t accepted;       /* accepted candidates                                 */
  int32_t producer_steps; /* drafter steps run                                   */
  int32_t published;      /* tokens published                                    */
} as2d_session_stats;

/* Run a session.  Producer service intervals are the drafter steps with their
   publication; verifier intervals are the as2d_verify_from_buffers calls
   (verification, read-back, alignment).  Blocking; synchronises both
   streams, which should be distinct non-default streams for the two sides to
   overlap on the GPU.  The drafter's capacity must leave room for one
   position per scripted token.  committed: host int32 [n_commit + AS2D_MAX_K + 1] or NULL
   receives the committed tokens; stats (required) the accounting.  Errors of
   either side stop the session and are returned. */
as2d_status as2d_session_run(const as2d_session_spec* spec, int32_t* committed,
                             as2d_session_stats* stats);

/* ---- Offline budget selection -----------------------------------------------
   (Section 3.3 "Device-profiled configuration": device cost profiles and
   development traces choose one fixed proposal budget b; App. B, Eq. for
   R(K), the per-position cost reduction of width K; App. D.2 "Fixed
   configurations and development splits": budgets ranked by pooled
   throughput.) */

/* Estimate the pooled committed tokens per second of every budget b in
   0..b_max on development traces.  Each trace is replayed with the alignment
   rules above: the producer's whole text is published before the first call
   (in AS2D_CBUF_BATCH-token batches), each call takes up to b candidates,
   the target commits the trace's reference text (accepting the longest
   matching prefix, then one token) until n_commit tokens are committed, and
   each call of k candidates is charged cost_us[k].
   cost_us: host double [AS2D_MAX_K + 1], mean call time by k (> 0).
   refs, prods: host int32, the traces' reference and producer texts
   concatenated, with lengths ref_len, prod_len host int32 [n_traces];
   ref_len[t] >= n_commit + b_max + 1.  window: the alignment search bound.
   Outputs (host): tok_s double [b_max + 1]; calls int32 [b_max + 1] (may be
   NULL), the pooled call counts; *best_b, the budget with the highest
   estimate (the smallest such b on ties). */
as2d_status as2d_budget_select(const double* cost_us, const int32_t* refs,
                               const int32_t* ref_len, const int32_t* prods,
                               const int32_t* prod_len, int32_t n_traces,
                               int32_t n_commit, int32_t window, int32_t b_max,
                               double* tok_s, int32_t* calls, int32_t* best_b);

/* Thread-local description of the last error ("" if none). */
const char* as2d_last_error(void);

#ifdef __cplusplus
}
#endif
#endif

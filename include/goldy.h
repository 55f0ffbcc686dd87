/*
 * goldy.h — C ABI of the concurrent-GEMM library (GO-Kernels + dynamic logic)
 * for one GB300 (sm_103a).
 *
 * The paper's problem (Sec. 4.1, Sec. 4.4): a set of independent GEMMs is
 * queued at once; the system picks how many run concurrently (the
 * concurrency degree, CD) and, for each GEMM, a kernel tuned for the
 * resources it will share at that CD (a "GO-Kernel"), then launches them.
 * This header splits that into
 *
 *   goldy_plan()  host only, integer work, no CUDA call: GEMM descriptors +
 *                 lookup table -> schedule (groups run one after another; in
 *                 a group, CD streams; per GEMM a kernel variant and a stream
 *                 slot).  The dynamic logic of Sec. 4.3 / Sec. 4.4.
 *   goldy_run()   asynchronous launch of a schedule on caller-owned streams
 *                 and caller-owned device buffers.  No allocation, no
 *                 synchronisation.  The GO-Kernels themselves (Sec. 4.2).
 *
 * Conventions for every entry point:
 *   - Return a goldy_status; nothing is thrown across the ABI.  On error the
 *     thread-local text of goldy_last_error() says why.
 *   - Pointers the caller passes stay owned by the caller.  Objects the
 *     library returns (goldy_lut, goldy_schedule, goldy_graph) are owned by
 *     the library and released with the matching *_free function.
 *   - Device pointers are plain CUDA device addresses on the current device;
 *     streams are cudaStream_t values passed as void*.
 *
 * Matrix layout (Sec. 2.1.2; transposes T1 = T2 = 0 in the K x N sense):
 *   A: M x K, row-major, element (i, k) at A[i*lda + k], bf16
 *   B: K x N, row-major, element (k, j) at B[k*ldb + j], bf16
 *   C: M x N, row-major, element (i, j) at C[i*ldc + j], fp32 or bf16
 *   C = A * B with fp32 accumulation; bf16 output is rounded to nearest even.
 */
#ifndef GOLDY_H_
#define GOLDY_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define GOLDY_ABI_VERSION 2

typedef enum goldy_status {
  GOLDY_OK = 0,
  GOLDY_ERR_INVALID_ARG = 1,   /* null pointer, bad size, bad stride, bad flags */
  GOLDY_ERR_UNSUPPORTED = 2,   /* valid request this build does not implement */
  GOLDY_ERR_LUT = 3,           /* lookup table missing, malformed or empty */
  GOLDY_ERR_CUDA = 4,          /* a CUDA runtime/driver call failed */
  GOLDY_ERR_TIMEOUT = 5,       /* a kernel gave up a bounded wait (see goldy_device_error) */
  GOLDY_ERR_NOMEM = 6          /* host allocation failed, or a caller buffer is too small */
} goldy_status;

typedef enum goldy_dtype { GOLDY_BF16 = 0, GOLDY_F32 = 1 } goldy_dtype;

/* One GEMM (Sec. 2.1.2), or a strided batch of equal-sized GEMMs (the
 * paper's B-GEMMs, Sec. 6.7): entry i computes C + i*stride_c = (A +
 * i*stride_a)(B + i*stride_b).  Sizes, leading dimensions and strides are in
 * elements.  Supported now: trans_a = trans_b = 0, a = b = GOLDY_BF16, c =
 * BF16 or F32, M, N, K >= 0, lda >= K, ldb >= N, ldc >= N, lda and ldb
 * multiples of 8 (16-byte rows for the tensor-memory-accelerator copies);
 * batch >= 1 (1: a plain GEMM, strides ignored); for batch > 1 the entries
 * do not overlap — stride_a >= M*lda, stride_b >= K*ldb, stride_c >= M*ldc —
 * and stride_a, stride_b are multiples of 8. */
typedef struct goldy_gemm_desc {
  int64_t M, N, K;
  int64_t lda, ldb, ldc;
  int32_t trans_a, trans_b;    /* the paper's T1, T2; only 0, 0 is supported */
  int32_t a_dtype, b_dtype, c_dtype;
  int32_t reserved;            /* must be 0 */
  int64_t batch;               /* strided batch entries, >= 1 */
  int64_t stride_a, stride_b, stride_c;
} goldy_gemm_desc;

typedef struct goldy_lut goldy_lut;
typedef struct goldy_schedule goldy_schedule;
typedef struct goldy_graph goldy_graph;

/* ---- planning policies (goldy_plan flags) -------------------------------
 * The comparison configurations of Sec. 5.5 through one schedule type:
 *   AUTO        the dynamic logic: preferred CD from the table, min(CD,
 *               available), heterogeneous grouping (Sec. 4.3, Sec. 6.7);
 *               then, in each wave (a group's members taken CD at a time,
 *               in launch order), a GEMM takes the kernel kind of the
 *               wave's largest GEMM (no K split, that kernel's grid cap)
 *               when the kind suits it — same C dtype, K no longer than the
 *               largest's, M >= 128 for a CTA-pair kind, M <= 2 x the tile
 *               rows for a transposed skinny-M kind, M >= 64 otherwise —
 *               so that a fused wave runs as fewer launches
 *   SEQUENTIAL  isolation-tuned kernels one after another ("sequential")
 *   DEFAULT     isolation-tuned kernels, every GEMM at once on its own stream
 *               ("default", the naive all-streams launch)
 *   GO          GO-Kernels for CD = n, every GEMM at once ("GO-Kernels")
 *   FORCE_CD    GO-Kernels at a fixed CD; put the CD in bits 8..15
 *               (GOLDY_PLAN_FORCE_CD | (cd << 8)) */
#define GOLDY_PLAN_AUTO 0
#define GOLDY_PLAN_SEQUENTIAL 1
#define GOLDY_PLAN_DEFAULT 2
#define GOLDY_PLAN_GO 3
#define GOLDY_PLAN_FORCE_CD 4
/* Launch-mode bit, combinable with any policy above.  FUSED: within each
 * group, the GEMMs that run at the same time (a "wave" of CD members) and
 * share a kernel kind and output dtype go into ONE persistent launch over the
 * concatenation of their tiles (at most 16 GEMMs per launch); its grid cap is
 * the sum of the members' caps.  A wave's launches carry launch priorities
 * ranked by their FLOPs, and the first wave's largest launch goes out first
 * (outside a stream capture the other streams also wait until all of its
 * CTAs have begun).  Groups are not separated by a join: the run forks once
 * and joins once, and a later group's launches take lower priorities, so they
 * fill the SMs an earlier group frees.  A fused run with
 * goldy_run_opts.inputs_ready = 1 goes out on streams[0] alone
 * instead, each wave's largest launch first, every launch overlapping the
 * previous one's tail (no fork, no join).  Without FUSED every GEMM is its own
 * launch on its slot's stream and the groups run one after another.  The plan
 * (groups, CDs, variants, slots) is the same, and so are the results, byte
 * for byte. */
#define GOLDY_PLAN_FUSED 0x10

#define GOLDY_MAX_GEMMS 64      /* GEMMs per plan */
#define GOLDY_MAX_STREAMS 16    /* concurrency degrees 1, 2, 4, 8, 16 (Sec. 4.3) */

/* ---- version / device ---------------------------------------------------- */

/* GOLDY_ABI_VERSION of the loaded library. */
int goldy_abi_version(void);

/* Text of the last error on this thread ("" if none).  Valid until the next
 * call into the library from the same thread. */
const char* goldy_last_error(void);

/* ---- kernel variant registry --------------------------------------------
 * A variant is one GO-Kernel configuration (Sec. 4.2): a tile shape and
 * shared-memory/tensor-memory footprint (kind), a split of the K loop, and a
 * resource constraint (RC) capping the persistent grid at the whole GPU, half
 * or a quarter of it (Sec. 4.2.1's GPU, GPU/2, GPU/4).  With a split S > 1
 * the S K-ranges of a tile are summed in split order 0 .. S-1 (in a cluster
 * of S CTAs, or by the last split to arrive, through the workspace; a CTA-pair
 * kind always through the workspace). */
typedef struct goldy_variant_info {
  int32_t id;
  int32_t kind;           /* tile/footprint family, 0 .. n_kinds-1 */
  int32_t mma_m;          /* rows of the tensor-core tile (128) */
  int32_t mma_n;          /* columns of the tensor-core tile */
  int32_t swap_ab;        /* 1: computes C^T = B^T A^T tiles (skinny M) */
  int32_t stages;         /* shared-memory pipeline depth */
  int32_t acc_stages;     /* accumulators held in tensor memory */
  int32_t tmem_cols;      /* tensor-memory columns allocated per CTA */
  int32_t smem_bytes;     /* dynamic shared memory per CTA */
  int32_t split_k;        /* K-loop split factor (1, 2, 4, 8) */
  int32_t rc_div;         /* grid cap = resident CTAs per SM * SMs / rc_div */
  int32_t ctas_per_sm;    /* CTAs per SM the footprint is sized for */
  int32_t cta_pair;       /* 2: tiles of 2 x 128 rows computed by a pair of CTAs
                             (one tcgen05 MMA across both SMs), else 1 */
  char name[32];
} goldy_variant_info;

/* Number of variant ids (ids are 0 .. count-1). */
int goldy_variant_count(void);

/* Describe variant `id`.  GOLDY_ERR_INVALID_ARG if id is out of range or out
 * is null. */
goldy_status goldy_variant_info_get(int id, goldy_variant_info* out);

/* ---- lookup table (the dynamic logic's profiled data, Sec. 4.3) ---------
 * File format (little-endian): magic "GOLDYLUT", u32 version = 1, u32 entry
 * count, u32 variant-id bound, u32 SM count of the profiling GPU, 8 zero
 * bytes; then 16-byte entries {u8 lm, ln, lk, out_dtype; u8 pref_cd; u8 flags;
 * u16 variant[5]} strictly sorted by (lm, ln, lk, out_dtype), where lm, ln,
 * lk are floor(log2) of M, N, K and variant[c] is the GO-Kernel for CD class
 * c in {1, 2, 4, 8, 16}; flags: how the bucket's GEMM runs with an
 * element-wise op of its output size (see goldy_corun_plan) — bit 0: at once
 * (else one after the other), bit 1: with the CD-2 GO-Kernel (else the CD-1
 * kernel), bits 2-3: the op's grid-cap divisor 1, 2 or 4 as 0, 1, 2; other
 * bits 0.  GOLDY_ERR_LUT if the data is malformed or empty. */
goldy_status goldy_lut_load(const char* path, goldy_lut** out);
goldy_status goldy_lut_from_memory(const void* data, size_t bytes, goldy_lut** out);
void goldy_lut_free(goldy_lut* lut);

/* Bucket key of one GEMM: (lm << 24) | (ln << 16) | (lk << 8) | c_dtype,
 * each log2 floored (0 for a size of 0) and clamped to 255; a batched GEMM
 * is bucketed by its rows over all entries (lm = floor log2(M * batch)). */
goldy_status goldy_bucket_key(const goldy_gemm_desc* d, uint32_t* key);

/* ---- planning (host only; makes no CUDA call) ---------------------------
 * Plan n (1 .. GOLDY_MAX_GEMMS) GEMMs with the policy in `flags`.
 * Deterministic: the schedule is a pure function of (descs, lut, flags).
 * GOLDY_ERR_INVALID_ARG for null pointers, n out of range, bad flags or a
 * descriptor violating the layout rules above; GOLDY_ERR_UNSUPPORTED for a
 * transposed operand or unsupported dtype. */
goldy_status goldy_plan(const goldy_gemm_desc* descs, int n, const goldy_lut* lut,
                        int flags, goldy_schedule** out);

/* ---- logistic-regression CD predictor (Sec. 4.3, Eq. 1) -----------------
 * The paper predicts each GEMM's preferred CD with a multi-class logistic
 * regression trained offline once per GPU.  Features (GOLDY_LR_FEATURES, in
 * this order): M (times the batch), N, K, then for each CD class c in (1, 2,
 * 4, 8, 16) three numbers of the table's GO-Kernel for the GEMM's bucket at
 * c: its CTAs of work (output tiles of all batch entries x split-K slices;
 * two CTAs per tile for a CTA-pair kernel), its CTAs resident per SM, and its waves (CTAs of work over
 * CTAs/SM x sm_count / grid-cap divisor, rounded up).  The model min-max
 * normalises them ((x - lo) / (hi - lo), 0 where hi == lo), scores each
 * class s_c = b_c + sum_j W[c][j] x_j (in j order, doubles, no fused
 * multiply-add), and predicts the class of largest score (= largest Eq. 1
 * probability; ties to the smaller CD).
 * Model file (little-endian): magic "GOLDYLRM", u32 version = 1, u32 feature
 * count = 18, u32 class count = 5, u32 SM count (> 0), 8 zero bytes; then
 * f64 lo[18], hi[18], W[5][18] (class-major), b[5]; all finite, hi >= lo.
 * GOLDY_ERR_LUT if malformed.  The library owns the object. */
#define GOLDY_LR_FEATURES 18
typedef struct goldy_predictor goldy_predictor;
goldy_status goldy_predictor_load(const char* path, goldy_predictor** out);
goldy_status goldy_predictor_from_memory(const void* data, size_t bytes, goldy_predictor** out);
void goldy_predictor_free(goldy_predictor* p);

/* The table entry a GEMM plans with (its bucket, or the nearest stored one):
 * preferred CD and the variant per CD class. */
goldy_status goldy_lut_lookup(const goldy_lut* lut, const goldy_gemm_desc* d, int* pref_cd, int variants[5]);

/* The predictor's raw (unnormalised) features of one GEMM against a table,
 * for an SM count (> 0).  Used to build the training set. */
goldy_status goldy_lr_features(const goldy_gemm_desc* d, const goldy_lut* lut, int sm_count,
                               double out[GOLDY_LR_FEATURES]);

/* Predicted preferred CD (1, 2, 4, 8 or 16) of one GEMM; probs (may be null)
 * receives Eq. 1's probability per CD class. */
goldy_status goldy_predict_cd(const goldy_predictor* p, const goldy_lut* lut, const goldy_gemm_desc* d,
                              int* cd, double probs[5]);

/* goldy_plan with the predictor (may be null: same as goldy_plan) supplying
 * the preferred CDs under GOLDY_PLAN_AUTO: a bucket's preference is the
 * smallest prediction over its GEMMs, and the CD run is still
 * min(preference, GEMMs available).  Kernels still come from the table.  The
 * forced policies ignore the predictor. */
goldy_status goldy_plan_ex(const goldy_gemm_desc* descs, int n, const goldy_lut* lut,
                           const goldy_predictor* predictor, int flags, goldy_schedule** out);

/* Explicit schedule (used by the offline profiler and for measuring any
 * chosen schedule): GEMM i runs in group group_of[i] (groups are run in
 * increasing order, ids 0 .. n_groups-1 all used), with variant
 * variant_of[i], on stream slot slot_of[i] (< GOLDY_MAX_STREAMS).  A group's
 * CD is its number of distinct slots.  flags: 0 or GOLDY_PLAN_FUSED (waves are
 * then the group's members taken CD at a time, in GEMM index order). */
goldy_status goldy_schedule_build(const goldy_gemm_desc* descs, int n, const int* group_of,
                                  const int* variant_of, const int* slot_of, int flags,
                                  goldy_schedule** out);

/* Sizes of a schedule.  workspace_bytes is the device workspace goldy_run
 * needs (split-K partial tiles and arrival counters, and for GOLDY_PLAN_FUSED
 * schedules of several GEMMs 8 bytes of unit counters per GEMM; 0 if none). */
goldy_status goldy_schedule_query(const goldy_schedule* s, int* n_gemms, int* n_groups,
                                  int* max_streams, size_t* workspace_bytes);

/* Placement of GEMM `gemm`: its group, variant, stream slot and its group's CD. */
goldy_status goldy_schedule_entry(const goldy_schedule* s, int gemm, int* group,
                                  int* variant, int* slot, int* cd);

/* Canonical bytes of the plan (little-endian u32 words): "GSCH", version 1,
 * n_gemms, n_groups, max_streams, flags; per group: cd, size, members in
 * launch order; per GEMM: group, variant, slot.  Writes at most `cap` bytes;
 * *size gets the full length (GOLDY_ERR_NOMEM if cap is too small). */
goldy_status goldy_schedule_serialize(const goldy_schedule* s, void* buf, size_t cap,
                                      size_t* size);

void goldy_schedule_free(goldy_schedule* s);

/* ---- execution ----------------------------------------------------------
 * Launch schedule `s`: A[i], B[i], C[i] are device pointers of GEMM i;
 * `workspace` is a device buffer of at least goldy_schedule_query's
 * workspace_bytes (may be null when that is 0), zero-filled by the caller
 * before its first use — the kernels leave it zero-filled after every
 * complete run; streams[0 .. n_streams-1] are CUDA streams with n_streams >=
 * max_streams.  Groups run in order (in GOLDY_PLAN_FUSED mode by launch
 * priority, see there); the run forks from streams[0] and joins back to it,
 * so work queued on streams[0] before the call happens before every GEMM and
 * work queued on streams[0] after it happens after all of them.  Slot k runs on streams[k].  Asynchronous: returns after launching;
 * no allocation, no synchronisation.  Errors: GOLDY_ERR_INVALID_ARG (null or
 * misaligned pointers, too few streams, workspace too small),
 * GOLDY_ERR_CUDA (launch failure).  A kernel that gave up a bounded wait
 * shows up later through goldy_device_error(); the outputs of that run are
 * then incomplete, and its workspace may hold non-zero split-K arrival or
 * unit counters: zero-fill the workspace again before the next run that uses
 * it. */
goldy_status goldy_run(const goldy_schedule* s, const void* const* A, const void* const* B,
                       void* const* C, void* workspace, size_t workspace_bytes,
                       void* const* streams, int n_streams);

/* Options of goldy_run_ex / goldy_graph_create_ex (all fields may be null).
 * ev_begin[i] / ev_end[i] (cudaEvent_t as void*, caller-created, one pair per
 * GEMM) are recorded on GEMM i's stream right before and right after its
 * kernel launch, so the caller can time each launch on the stream it runs on.
 * Inside a graph capture they become event-record nodes of the graph. */
typedef struct goldy_run_opts {
  void* const* ev_begin;
  void* const* ev_end;
  /* Optional device buffer of unsigned 64-bit words for a phase trace: every
   * CTA of every GO-Kernel launch writes 16 words at trace[cta * 16 + k]
   * (k: 0 entry, 1 set-up done and the epilogue past the wait for the
   * previous kernel, 2 first TMA load, 3 first full stage seen by
   * the MMA thread, 4 first accumulator committed, 5 first accumulator seen
   * by the epilogue, 6 split-K partial stored, 7 split-K arrival counted,
   * 8 first unit stored, 9 exit, 10 set-up done before waiting for the
   * previous kernel on the stream, 11 producer started — %globaltimer
   * nanoseconds; 12 the launch's grid size; 13 the CTA's index in its launch;
   * 14 units this CTA processed; 15 SM id).  The launches of one run use
   * consecutive regions in launch order (launch j starts after the CTAs of
   * launches 0 .. j-1); a launch that does not fit in the trace_ctas CTAs
   * left is not traced.  Null: no tracing. */
  void* trace;
  size_t trace_ctas;
  /* 0 (default): each GO-Kernel launch may begin its set-up (barriers, tensor
   * memory, descriptor prefetch) while the previous kernel on its stream is
   * still running — programmatic dependent launch; the kernel waits for that
   * kernel to complete before it touches global memory, so results and
   * stream order are unchanged.  1: plain serialised launches. */
  int32_t serial_launch;
  /* 0 (default): as above.  1: the caller asserts that no kernel enqueued
   * before this run (on its streams) writes any A or B of the run.  Each
   * GO-Kernel's load and MMA roles then start as soon as its CTAs are
   * resident, while the previous kernel on the stream may still be running
   * (reading A and B, filling shared and tensor memory); the epilogue still
   * waits for that kernel to complete before it writes C or the workspace.
   * Results are unchanged when the assertion holds; a violated assertion
   * (an earlier kernel producing A or B) gives wrong results.  The bounded
   * waits of the load and MMA roles then also cover the previous kernel's
   * remaining time.  No effect with serial_launch = 1. */
  int32_t inputs_ready;
  /* Limit of every bounded wait inside the GO-Kernels, in microseconds
   * (0: the default of 2 seconds).  A wait that runs out sets the error word
   * (goldy_device_error) and the kernel returns. */
  uint32_t wait_limit_us;
  /* Test hook, 0 in normal use.  1: in the run's first GO-Kernel launch, CTA
   * 0 never fills its first shared-memory stage (no copy is issued), so that
   * the MMA thread's bounded wait for it runs out: the launch returns with
   * the error word set to 2 (an MMA-thread wait gave up) and the outputs of
   * that launch are incomplete.  Used with a short wait_limit_us to test the
   * timeout path without faulting anything. */
  int32_t test_stall_first_stage;
} goldy_run_opts;

/* goldy_run with options; opts may be null (then identical to goldy_run). */
goldy_status goldy_run_ex(const goldy_schedule* s, const void* const* A, const void* const* B,
                          void* const* C, void* workspace, size_t workspace_bytes,
                          void* const* streams, int n_streams, const goldy_run_opts* opts);

/* Prepared run: record goldy_run_ex(...) with these exact pointers and
 * streams once — tensor maps encoded, kernel parameter blocks built, grids and
 * cluster shapes fixed, fork/join events owned by the object — so that
 * goldy_exec_launch replays it with plain launch calls on the same streams.
 * On this platform a replay costs about half of a one-kernel CUDA graph
 * launch.  Nothing is launched by goldy_exec_create; the buffers and streams
 * must outlive the object.  Not thread-safe per object. */
typedef struct goldy_exec goldy_exec;
goldy_status goldy_exec_create(const goldy_schedule* s, const void* const* A, const void* const* B,
                               void* const* C, void* workspace, size_t workspace_bytes,
                               void* const* streams, int n_streams, const goldy_run_opts* opts,
                               goldy_exec** out);
/* Enqueue a prepared run (asynchronous, no allocation). */
goldy_status goldy_exec_launch(const goldy_exec* e);
void goldy_exec_free(goldy_exec* e);

/* Device time of prepared runs replayed back to back: `warmup` untimed
 * replays, then `reps` replays timed by CUDA events on the first stream
 * (replay k uses execs[k % n]: rotate copies of the inputs past the L2).  All
 * n runs must share their first stream and partition.  Synchronises on the
 * end event; *ms_per_rep = elapsed / reps.  Events live in the runs'
 * partition, so this also times work inside an SM partition. */
goldy_status goldy_exec_time(const goldy_exec* const* execs, int n, int warmup, int reps, float* ms_per_rep);

/* ---- a GEMM co-scheduled with a non-GEMM kernel (Sec. 7.1) --------------
 * The paper co-runs a GEMM with an element-wise add of the GEMM's output size
 * (2 kernels at once) and finds concurrency worth restricting for
 * memory-bound GEMMs.  The non-GEMM here is Z = X + Y over n contiguous
 * elements of `dtype` (bf16: each element widened to fp32, added in IEEE
 * fp32 with round-to-nearest-even, rounded back to bf16 RNE; fp32: one IEEE
 * fp32 addition), by a persistent grid-stride kernel whose grid is capped at
 * 8 CTAs/SM x SMs / rc_div (rc_div 1, 2 or 4: GPU, GPU/2, GPU/4).
 *
 * Policies (goldy_corun_plan):
 *   GOLDY_PLAN_SEQUENTIAL  isolation-tuned GEMM kernel, then the add, one stream
 *   GOLDY_PLAN_DEFAULT     isolation-tuned GEMM kernel and the add (whole-GPU
 *                          grid) at once on two streams
 *   GOLDY_PLAN_GO          the table's CD-2 GO-Kernel and the add capped at
 *                          GPU/2, at once
 *   GOLDY_PLAN_AUTO        the configuration the table entry's flags record
 *                          (profiled: the fastest of running at once with the
 *                          CD-1 or CD-2 kernel and the op capped at GPU,
 *                          GPU/2 or GPU/4, taken only when it beats one after
 *                          the other by >= 5%), else SEQUENTIAL — concurrency
 *                          restricted where it does not pay.
 * The table's kernels are those of the GEMM's bucket (see goldy_lut_lookup). */
typedef struct goldy_ewise_desc {
  int64_t n;        /* elements (>= 0) */
  int32_t dtype;    /* GOLDY_BF16 or GOLDY_F32, for X, Y and Z */
  int32_t reserved; /* must be 0 */
} goldy_ewise_desc;
typedef struct goldy_corun goldy_corun;
goldy_status goldy_corun_plan(const goldy_gemm_desc* gemm, const goldy_ewise_desc* ew, const goldy_lut* lut,
                              int policy, goldy_corun** out);
/* concurrent: 1 if the two kernels run at once (needs 2 streams); the GEMM's
 * variant; the add's grid-cap divisor; device workspace bytes (split-K). */
goldy_status goldy_corun_query(const goldy_corun* c, int* concurrent, int* gemm_variant, int* add_rc_div,
                               size_t* workspace_bytes);
/* Enqueue: the GEMM C = A B on streams[0]; the add on streams[1] (forked
 * from and joined back into streams[0]) when concurrent, else on streams[0]
 * after the GEMM.  X, Y, Z: device arrays of n elements; the vector path
 * needs them 16-byte aligned (others take a scalar path).  Asynchronous. */
goldy_status goldy_corun_run(const goldy_corun* c, const void* A, const void* B, void* C, void* workspace,
                             size_t workspace_bytes, const void* X, const void* Y, void* Z, void* const* streams,
                             int n_streams);
/* The same, recorded once as a prepared run (see goldy_exec_create). */
goldy_status goldy_corun_exec_create(const goldy_corun* c, const void* A, const void* B, void* C, void* workspace,
                                     size_t workspace_bytes, const void* X, const void* Y, void* Z,
                                     void* const* streams, int n_streams, goldy_exec** out);
void goldy_corun_free(goldy_corun* c);

/* The element-wise add alone on one stream (rc_div 1, 2 or 4). */
goldy_status goldy_ewise_add(const void* X, const void* Y, void* Z, int64_t n, int dtype, int rc_div, void* stream);

/* ---- SM partitions (CU-Partition, Sec. 6.9; GPU-Quarter/Half, Sec. 7.4) -----------
 * A partition is a CUDA green context owning a subset of the GPU's SMs plus
 * n_streams (1 .. GOLDY_MAX_STREAMS) non-blocking streams in it; kernels
 * enqueued on those streams run on the partition's SMs only.  min_sms <= 0
 * or >= the device's SMs gives the whole device as a partition; otherwise the
 * driver rounds min_sms up to its partition granularity (query the actual
 * count).  Passing a partition's streams to goldy_run / goldy_run_ex /
 * goldy_exec_create / goldy_graph_create(_ex) / goldy_graph_launch runs the
 * schedule inside the partition: grid caps are computed from the partition's
 * SM count, and the library makes the partition's context current on the
 * calling thread for the duration of each call (device memory of the
 * device's primary context stays valid).  GOLDY_ERR_UNSUPPORTED if the
 * driver has no green contexts or cannot split off such a partition.  Free
 * every exec and graph that uses a partition before the partition. */
typedef struct goldy_partition goldy_partition;
goldy_status goldy_partition_create(int min_sms, int n_streams, goldy_partition** out);
/* SM count, and the first n (<= n_streams) streams (CUstream handles). */
goldy_status goldy_partition_query(const goldy_partition* p, int* sm_count, void** streams, int n);
void goldy_partition_free(goldy_partition* p);

/* Capture goldy_run(...) with these exact pointers into a CUDA graph, for
 * replay with one launch (the closest host-side analogue of the command
 * processor dispatching a whole set).  The streams must be idle.  The graph
 * owns copies of all launch parameters; the buffers must outlive it. */
goldy_status goldy_graph_create(const goldy_schedule* s, const void* const* A,
                                const void* const* B, void* const* C, void* workspace,
                                size_t workspace_bytes, void* const* streams, int n_streams,
                                goldy_graph** out);
/* goldy_graph_create with run options (event hooks captured into the graph). */
goldy_status goldy_graph_create_ex(const goldy_schedule* s, const void* const* A,
                                   const void* const* B, void* const* C, void* workspace,
                                   size_t workspace_bytes, void* const* streams, int n_streams,
                                   const goldy_run_opts* opts, goldy_graph** out);
/* Launch a captured graph on `stream` (asynchronous). */
goldy_status goldy_graph_launch(const goldy_graph* g, void* stream);
void goldy_graph_free(goldy_graph* g);

/* One GEMM with GO-Kernel variant `variant`, for callers that cannot allocate
 * device memory (the paper has no counterpart; this is a service of this
 * library).  goldy_run needs a caller workspace for split-K variants; callers
 * held to a fixed memory budget, plugins inside a framework that owns all
 * device allocations, and paths where cudaMalloc's implicit synchronisation
 * is unacceptable cannot provide one.  Here the split-K scratch is a fixed
 * 32 MiB device array compiled into the library (one per GPU that loads it,
 * held until exit); nothing is allocated.  Launches on `stream`
 * (cudaStream_t as void*, may be null; a stream of an SM partition runs the
 * GEMM inside the partition, as goldy_run does) and returns without
 * synchronising.  A, B, C, desc: as for goldy_run (16-byte aligned A and B).
 * Errors: GOLDY_ERR_INVALID_ARG for a bad descriptor, variant or pointer, or
 * when the GEMM would need more than the 32 MiB scratch (the message gives the
 * size); GOLDY_ERR_CUDA for a failed launch.  The first call on a device looks
 * up the scratch's device address (cudaGetSymbolAddress, which may load
 * device code) and keeps it for the life of the process: make that call
 * before any stream capture, and do not call this entry point on a device
 * after cudaDeviceReset.  All calls share the scratch: calls whose kernels
 * overlap on the GPU race and give wrong results, so serialise them (one
 * stream, or events). */
goldy_status goldy_gemm_noalloc(const goldy_gemm_desc* desc, int variant, const void* A,
                                const void* B, void* C, void* stream);

/* Error word the kernels set when a bounded wait gives up (0 = none; the
 * first failure wins): 1 a load-role wait, 2 an MMA-thread wait, 3 an
 * epilogue wait, 4 a split-K cluster-exchange wait.  Reads it synchronously
 * on the current device and, if `clear`, resets it.  After a non-zero code,
 * zero-fill the workspace of the failed run before reusing it (goldy_run). */
goldy_status goldy_device_error(int* code, int clear);

/* SM count and CTAs of variant `variant_id` resident per SM on the current
 * device (occupancy query, no launch). */
goldy_status goldy_device_info(int variant_id, int* sm_count, int* ctas_per_sm);

#ifdef __cplusplus
}
#endif

#endif /* GOLDY_H_ */

/*
 * trident_scm.h -- C ABI of the Specialization Cache Module (SCM) library.
 *
 * The SCM is the paper's central artifact (Trident, §3.1 and Fig. 1c): an ordered
 * set of versions, each a guard predicate G_i paired with the computation P_i captured
 * under it, plus a dispatcher that runs the first P_i whose G_i holds (§3.2, Algorithm 1).
 * A cache hit stays in native code from guard evaluation through argument preparation
 * and the kernel launch; only a miss leaves the library, through a compile hook (§3.5).
 *
 * In this library P_i is a hand-written sm_103a CUDA kernel for one step of an LLM
 * decoder layer's memory-bound chain (fused residual-add + RMSNorm, per-head q/k
 * RMSNorm, RoPE with KV-cache append, SwiGLU, or the whole chain in one launch).
 * The layer math is not given by the paper, which runs these operators inside the
 * Qwen3-8B / DeepSeek-V2-Lite decode loops it evaluates (§4.1); the formulas each op
 * computes are stated below, next to the op.
 *
 * Conventions for every entry point:
 *   - Tensors are described, never owned: the caller owns every buffer and the stream.
 *   - Strides and shapes are in ELEMENTS. Pointers are device addresses for tensors
 *     whose device field is >= 0.
 *   - Return values are trident_status codes. Values >= 0 are not errors. A miss is
 *     never an error code, and an error never triggers the compile hook (§3.2, §3.4,
 *     §3.5: "miss" and "error" stay distinct).
 *   - On an error, trident_scm_last_error() returns a thread-local message.
 *   - All functions are thread-safe unless stated otherwise. The hit path of
 *     trident_scm_invoke takes no lock and allocates nothing.
 */
#ifndef TRIDENT_SCM_H
#define TRIDENT_SCM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define TRIDENT_ABI_VERSION 4
#define TRIDENT_MAX_TENSORS 20
#define TRIDENT_MAX_FIXED 8
/* out_selected value for a sequence element that was not run (trident_scm_invoke_seq). */
#define TRIDENT_NOT_RUN (-2)

/* ---------------------------------------------------------------- status codes */
typedef enum trident_status {
  TRIDENT_OK = 0,             /* hit: version *out_selected ran (Algorithm 1, return o)      */
  TRIDENT_MISS_HANDLED = 1,   /* every guard failed; the compile hook ran and succeeded     */
  TRIDENT_MISS = 2,           /* every guard failed and no hook ran (Algorithm 1, MISS)     */
  TRIDENT_ERR_INVALID = -1,   /* malformed arguments, descriptor or launch precondition     */
  TRIDENT_ERR_CUDA = -2,      /* a CUDA call failed (launch, allocation, copy)              */
  TRIDENT_ERR_HOOK = -3,      /* the compile hook returned non-zero                         */
  TRIDENT_ERR_CAPACITY = -4,  /* the version table is full                                  */
  TRIDENT_ERR_STATE = -5      /* the call is not allowed in this mode (e.g. dry-run launch) */
} trident_status;

/* ---------------------------------------------------------------- dtypes */
typedef enum trident_dtype {
  TRIDENT_BF16 = 1,  /* 2 bytes */
  TRIDENT_FP16 = 2,  /* 2 bytes */
  TRIDENT_FP32 = 3,  /* 4 bytes */
  TRIDENT_I32 = 4,   /* 4 bytes */
  TRIDENT_I64 = 5,   /* 8 bytes */
  TRIDENT_U8 = 6     /* 1 byte (masks: 0 false, non-zero true) */
} trident_dtype;

/* ---------------------------------------------------------------- operations
 * Each op has a fixed tensor order ("slots"). T is the token count; "act" is the
 * activation dtype (bf16, fp16, or fp32 where noted). All float math is fp32.
 *
 * TRIDENT_OP_ADD_RMSNORM (5 tensors; act = bf16 | fp16 | fp32; rank 2 [T,H] or 3 [B,S,H], T = B*S)
 *   0 x [T,H] act   1 r [T,H] act   2 gamma [H] fp32   3 y [T,H] act (out)   4 r_out [T,H] act (out)
 *   s = x + r;  r_out = round(s);  y = round(s * rsqrt(mean(s^2) + eps) * gamma)
 *   In place: y may be x and r_out may be r (same pointer, shape and strides).
 *
 * TRIDENT_OP_RMSNORM (3 tensors; act = bf16 | fp16 | fp32; rank 2 [T,H] or 3 [B,S,H], T = B*S)
 *   0 x [T,H] act   1 gamma [H] fp32   2 y [T,H] act (out)
 *   y = round(x * rsqrt(mean(x^2) + eps) * gamma) -- the paper's running example operator,
 *   rms_norm (§2.3, Fig. 1). In place: y may be x.
 *
 * Pointwise operators of the paper's kernel benchmark (§4.1, §4.2; FlagGems-style), over
 * rows [T,W] or [B,S,W] (T = B*S), act = bf16 | fp16 | fp32, W the version's fixed size:
 * TRIDENT_OP_SILU (2 tensors)         0 x, 1 y (out):  y = round(x / (1 + exp(-x)))
 * TRIDENT_OP_ADD (3 tensors)          0 a, 1 b, 2 y (out):  y = round(a + b), summed in fp32
 * TRIDENT_OP_NEG (2 tensors)          0 x, 1 y (out):  y = -x
 * TRIDENT_OP_MASKED_FILL (3 tensors)  0 x, 1 mask [T,W] u8, 2 y (out):
 *                                     y = mask != 0 ? round(args.scalar) : x
 *   In place: y may be x (or a or b for ADD).
 *
 * TRIDENT_OP_ROPE_KV (6 tensors; act = bf16 | fp16)
 *   0 q [T,Hq,D] act (in/out)  1 k [T,Hkv,D] act  2 v [T,Hkv,D] act  3 pos [T] i32
 *   4 k_cache [Hkv,S,D] act (out)  5 v_cache [Hkv,S,D] act (out)
 *   Rotate-half RoPE with inv_freq_i = theta^(-2i/D), i < D/2, angle a = pos * inv_freq_i:
 *     x'_i = x_i cos a - x_{i+D/2} sin a,   x'_{i+D/2} = x_{i+D/2} cos a + x_i sin a.
 *   q is rotated in place; k_cache[h, pos[t], :] = round(rope(k[t,h,:]));
 *   v_cache[h, pos[t], :] = v[t,h,:] (bit copy). Positions in one call must be distinct.
 *   A position outside [0,S) is skipped for that token (q, k and v untouched) and sets
 *   bit TRIDENT_DEVERR_POS in the device status word (trident_scm_device_status).
 *
 * TRIDENT_OP_QKNORM_ROPE_KV (8 tensors; act = bf16 | fp16)
 *   slots 0-5 as ROPE_KV, 6 gamma_q [D] fp32, 7 gamma_k [D] fp32.
 *   Before the rotation each q head and each k head is RMS-normalised over its D
 *   elements and scaled by gamma_q / gamma_k (eps from args); the result is not rounded
 *   between the norm and the rotation.
 *
 * TRIDENT_OP_SWIGLU (3 tensors; act = bf16 | fp16 | fp32; rank 2 [T,I] or 3 [B,S,I])
 *   0 g [T,I] act  1 u [T,I] act  2 out [T,I] act (out)
 *   out = round(g / (1 + exp(-g)) * u).  In place: out may be g or u.
 *
 * TRIDENT_OP_LAYER_CHAIN (18 tensors; act = bf16 | fp16): one decoder layer's non-GEMM chain
 *   0 h [T,H]  1 r0 [T,H]  2 gamma_attn [H]  3 x1 [T,H] out  4 r1 [T,H] out
 *   5 q [T,Hq,D] in/out  6 k [T,Hkv,D]  7 v [T,Hkv,D]  8 pos [T] i32
 *   9 k_cache [Hkv,S,D] out  10 v_cache [Hkv,S,D] out
 *   11 attn_out [T,H]  12 gamma_mlp [H]  13 x2 [T,H] out  14 r2 [T,H] out
 *   15 g [T,I]  16 u [T,I]  17 o [T,I] out
 *   = ADD_RMSNORM(h, r0, gamma_attn -> x1, r1); ROPE_KV(q, k, v, pos, caches);
 *     ADD_RMSNORM(attn_out, r1, gamma_mlp -> x2, r2); SWIGLU(g, u -> o).
 *   The second norm reads r1 as rounded to act. In place: x1 = h, r1 = r0, x2 = attn_out,
 *   r2 = r1, o = g or o = u.
 *
 * TRIDENT_OP_LAYER_CHAIN_QKNORM (20 tensors): LAYER_CHAIN with QKNORM_ROPE_KV instead of
 *   ROPE_KV; 18 gamma_q [D] fp32, 19 gamma_k [D] fp32.
 */
typedef enum trident_op {
  TRIDENT_OP_ADD_RMSNORM = 1,
  TRIDENT_OP_ROPE_KV = 2,
  TRIDENT_OP_QKNORM_ROPE_KV = 3,
  TRIDENT_OP_SWIGLU = 4,
  TRIDENT_OP_LAYER_CHAIN = 5,
  TRIDENT_OP_LAYER_CHAIN_QKNORM = 6,
  TRIDENT_OP_RMSNORM = 7,
  TRIDENT_OP_SILU = 8,
  TRIDENT_OP_ADD = 9,
  TRIDENT_OP_NEG = 10,
  TRIDENT_OP_MASKED_FILL = 11
} trident_op;

/* Layout class of an argument tuple (guard field, §2.2.1 "shape-related metadata").
 * Over the op's activation tensors (not gamma, pos or the caches):
 *   every tensor needs unit element stride and packed inner dims, else the tuple has
 *   no layout class and matches no version;
 *   CONTIG      every tensor's row stride equals its row width (a tensor with one row
 *               always counts as contiguous, as torch's is_contiguous does);
 *   ROWSTRIDED  not CONTIG, and every row stride is >= the row width.
 * A version's layout is CONTIG or ROWSTRIDED (exact match) or ANY (either class). */
typedef enum trident_layout {
  TRIDENT_LAYOUT_CONTIG = 0,
  TRIDENT_LAYOUT_ROWSTRIDED = 1,
  TRIDENT_LAYOUT_ANY = 2
} trident_layout;

/* Kernel family of a version. AUTO picks VECTOR when the version allows it. */
typedef enum trident_variant {
  TRIDENT_VARIANT_AUTO = 0,
  TRIDENT_VARIANT_GENERIC = 1,  /* scalar element access: any alignment, any row width  */
  TRIDENT_VARIANT_VECTOR = 2    /* 128/256-bit accesses: align_bytes 16, supported sizes */
} trident_variant;

/* Bits of the device status word. */
#define TRIDENT_DEVERR_POS 0x1u   /* a RoPE/KV position was outside [0, S) */
#define TRIDENT_DEVERR_TIMEOUT 0x2u /* a kernel's bounded wait for its own bulk copies ran
                                       out; that block's outputs were not written */

/* Option flags of trident_scm_create. */
#define TRIDENT_OPT_DRY_RUN 0x1        /* no CUDA at all: invoke selects and calls the hook,
                                          but launches nothing (host-only testing) */
#define TRIDENT_OPT_NO_ALIAS_CHECK 0x2 /* skip the output-overlap launch precondition */
#define TRIDENT_OPT_PDL 0x4            /* launch with programmatic stream serialisation */
#define TRIDENT_OPT_TIMING 0x8         /* record host ns per hit (trident_scm_host_times) */
#define TRIDENT_OPT_FAIL_LAUNCHES 0x10 /* fault injection on the host, for tests: every launch
                                          step of a hit reports ERR_CUDA without launching */
#define TRIDENT_OPT_NO_STEP_REPLAY 0x20 /* invoke_step never replays a stored chunk */
#define TRIDENT_OPT_TEST_WAIT_TIMEOUT 0x40 /* for tests of the device-side timeout path: the
                                          bulk-copy add+RMSNorm kernel gives up its first
                                          wait for its copies at once (0 polls), so every
                                          block takes the timeout path -- sets
                                          TRIDENT_DEVERR_TIMEOUT, drains its copies with the
                                          full bounded wait and returns without writing */

/* ---------------------------------------------------------------- structs */
/* Caller-owned tensor descriptor (DLPack-like, §3.4: tensors cross the boundary as
 * descriptors). 88 bytes. */
typedef struct trident_tensor {
  void* data;            /* device address (or host address if device < 0); may be NULL
                            only when the tensor has no elements */
  int64_t shape[4];      /* first ndim entries used, each >= 0 */
  int64_t stride[4];     /* elements, each >= 0 */
  int32_t dtype;         /* trident_dtype */
  int32_t ndim;          /* 1..4 */
  int32_t device;        /* CUDA ordinal, or -1 for host memory (matches no version) */
  int32_t reserved;
} trident_tensor;

/* One invocation's argument tuple: the op, its tensors in slot order, and scalars. */
typedef struct trident_args {
  int32_t op;            /* trident_op */
  int32_t ntensors;      /* must equal the op's slot count */
  double eps;            /* RMSNorm epsilon (runtime scalar, not guarded), must be >= 0 */
  double rope_theta;     /* RoPE base; a specialised constant (guarded by equality, §3.3) */
  double scalar;         /* MASKED_FILL's fill value (runtime scalar, not guarded) */
  int32_t flags;         /* reserved, must be 0 */
  int32_t reserved;
  trident_tensor t[TRIDENT_MAX_TENSORS];
} trident_args;

/* Descriptor of one version (specialisation). register_spec copies it. */
typedef struct trident_spec_desc {
  int32_t op;                       /* trident_op                                        */
  int32_t dtype;                    /* activation dtype                                  */
  int32_t rank;                     /* rank of slot 0 (2 or 3 for the norms, SWIGLU and
                                       the pointwise ops,
                                       3 for ROPE ops, 2 for the chains)                  */
  int32_t layout;                   /* trident_layout                                    */
  int64_t fixed[TRIDENT_MAX_FIXED]; /* fixed sizes: ADD_RMSNORM, RMSNORM {H}; SWIGLU {I};
                                       SILU, ADD, NEG, MASKED_FILL {W};
                                       ROPE ops {Hq, Hkv, D, S};
                                       chains {H, Hq, Hkv, D, S, I}; unused entries 0    */
  int64_t tok_lo, tok_hi;           /* inclusive token-count bucket, 1 <= lo <= hi       */
  int32_t align_bytes;              /* 16: every pointer and every outer stride 16-byte
                                       aligned (positions excepted: read per element);
                                       or the element size (no extra requirement)        */
  int32_t device;                   /* CUDA ordinal; must equal the SCM's device         */
  int32_t variant;                  /* trident_variant                                   */
  int32_t reserved;
  double rope_theta;                /* ROPE ops and chains: guarded constant; else 0     */
} trident_spec_desc;

struct trident_scm; /* the SCM handle (trident_scm_t below) */

/* ---------------------------------------------------------------- structured arguments
 * §3.3 of the paper: the boundary sees the source function's structured arguments (tuples
 * of tensors, scalars, None); each version's recipe binds them to a logical input tree,
 * guards address values by their path in that tree, and only after the guards hold are the
 * leaves the version consumes taken out, in the tree's preorder ("exporter order").
 *
 * A call's arguments are one array of nodes: nodes[0 .. nargs-1] are the top-level
 * parameters in source order; a tuple's n children are nodes[first .. first+n-1], and
 * first > the tuple's own index (children come after their parent, so the tree has no
 * cycles). At most TRIDENT_TREE_MAX_NODES nodes and depth TRIDENT_TREE_MAX_DEPTH. */
#define TRIDENT_TREE_MAX_NODES 4096
#define TRIDENT_TREE_MAX_DEPTH 16
typedef enum trident_node_kind {
  TRIDENT_NODE_NONE = 0,      /* Python None                                             */
  TRIDENT_NODE_TENSOR = 1,    /* t: a tensor descriptor                                  */
  TRIDENT_NODE_DLTENSOR = 2,  /* dl: a DLPack DLTensor (the layout shared by DLPack 0.6
                                 to 1.x: data, device {type, id}, ndim, dtype {code,
                                 bits, lanes}, shape, strides (NULL = compact), byte
                                 offset). Accepted: CUDA or CPU devices; bf16, fp16,
                                 fp32, int32, int64, uint8 and bool, one lane.          */
  TRIDENT_NODE_TUPLE = 3,     /* n children at nodes[first ...]                          */
  TRIDENT_NODE_INT = 4,       /* i                                                       */
  TRIDENT_NODE_FLOAT = 5      /* f                                                       */
} trident_node_kind;

typedef struct trident_node {
  int32_t kind;       /* trident_node_kind                    */
  int32_t n;          /* TUPLE: number of children            */
  int32_t first;      /* TUPLE: index of the first child      */
  int32_t reserved;   /* 0                                    */
  int64_t i;          /* INT                                  */
  double f;           /* FLOAT                                */
  const void* dl;     /* DLTENSOR: a DLTensor*                */
  trident_tensor t;   /* TENSOR                               */
} trident_node;

/* A version's recipe: a pattern over the call's tree, in the same array form. Each
 * pattern node requires the argument at the same path to have its kind (a TENSOR pattern
 * accepts TENSOR and DLTENSOR nodes; a TUPLE pattern requires exactly n children) and
 * says what the version does with it (bind):
 *   TENSOR: the op slot (0 .. ntensors-1) the leaf fills, or TRIDENT_BIND_UNUSED;
 *   INT / FLOAT: TRIDENT_BIND_CONST (a guarded constant: the value must equal i / f),
 *     TRIDENT_BIND_EPS, _THETA or _SCALAR (the value becomes that argument of the op), or
 *     TRIDENT_BIND_UNUSED (any value);
 *   NONE, TUPLE: bind is ignored.
 * Every slot of the version's op is bound by exactly one TENSOR pattern node. eps,
 * rope_theta and scalar not bound from the tree take the recipe's values. */
#define TRIDENT_BIND_UNUSED (-1)
#define TRIDENT_BIND_CONST (-2)
#define TRIDENT_BIND_EPS (-3)
#define TRIDENT_BIND_THETA (-4)
#define TRIDENT_BIND_SCALAR (-5)
typedef struct trident_recipe_node {
  int32_t kind;       /* trident_node_kind (not DLTENSOR)      */
  int32_t n;          /* TUPLE: number of children             */
  int32_t first;      /* TUPLE: index of the first child       */
  int32_t bind;       /* see above                             */
  int64_t i;          /* INT with TRIDENT_BIND_CONST           */
  double f;           /* FLOAT with TRIDENT_BIND_CONST         */
} trident_recipe_node;

typedef struct trident_recipe {
  int32_t nargs;                      /* top-level parameters: nodes[0 .. nargs-1]  */
  int32_t nnodes;
  const trident_recipe_node* nodes;   /* copied by register_tree_spec               */
  double eps, rope_theta, scalar;     /* values not bound from the tree             */
} trident_recipe;

/* Compile hook of invoke_tree (see trident_scm_set_tree_hook). */
typedef int32_t (*trident_tree_hook)(void* user, struct trident_scm* scm, const trident_node* nodes,
                                     int32_t nargs, int32_t nnodes, void* stream,
                                     int32_t* out_registered);

typedef struct trident_scm_options {
  int32_t device;        /* CUDA ordinal the SCM launches on (ignored for DRY_RUN) */
  int32_t max_specs;     /* capacity of the version table, 1..4096 (0 = 256)       */
  int32_t flags;         /* TRIDENT_OPT_*                                           */
  int32_t timing_ring;   /* samples kept by TRIDENT_OPT_TIMING (0 = 65536)          */
} trident_scm_options;

typedef struct trident_scm_stats_t {
  uint64_t invokes;         /* calls of invoke (each element of invoke_seq counts)  */
  uint64_t hits;            /* guard hits that launched (or would, in dry-run)       */
  uint64_t misses;          /* calls where every guard failed                        */
  uint64_t hook_calls;      /* misses that called the hook                           */
  uint64_t hook_failures;   /* hook calls that returned non-zero                     */
  uint64_t hook_registered; /* versions registered from inside a hook                */
  uint64_t err_invalid;     /* ERR_INVALID returns (validation or precondition)      */
  uint64_t err_cuda;        /* ERR_CUDA returns                                      */
  uint64_t guard_evals;     /* versions whose guard was evaluated                    */
  int32_t num_specs;        /* versions in the current table                         */
  int32_t reserved;
  uint64_t fused_launches;  /* invoke_step launches that ran several calls at once   */
  uint64_t fused_calls;     /* calls run by those launches                           */
  uint64_t step_replays;    /* calls of fused chunks relaunched from the replay cache
                               (counted in invokes, hits and fused_calls as well; no
                               guard is evaluated for them)                          */
} trident_scm_stats_t;

typedef struct trident_scm trident_scm_t; /* opaque; owns the table, kernels and device state */

/* Compile hook, called by invoke only on a miss (§3.5: an empty SCM takes the same
 * path on its first call). The hook must produce the result of this call (§3.5: the
 * call that triggered compilation returns the captured result), for example by
 * registering a version and re-invoking, or by invoking a second SCM. It may call
 * register_spec and invoke on `scm` (a miss inside a hook does not call the hook
 * again). It writes the index it registered, or -1, to *out_registered, and returns
 * 0 on success or non-zero on failure (invoke then returns TRIDENT_ERR_HOOK). */
typedef int32_t (*trident_compile_hook)(void* user, trident_scm_t* scm, const trident_args* args,
                                        void* stream, int32_t* out_registered);

/* ---------------------------------------------------------------- entry points */

/* Version of this ABI (TRIDENT_ABI_VERSION). §3.4: one packed ABI is the common boundary
 * between the dispatcher and its callers, exposed under one stable entry symbol; a caller
 * built against another layout of the structs below checks this number before its first
 * call instead of passing misread arguments. Needs no GPU; never fails. */
int32_t trident_abi_version(void);

/* Creates an empty SCM (§3.5: an empty SCM takes the miss path first).
 * opt may be NULL (device 0, 256 versions, no flags). hook and user may be NULL.
 * Without TRIDENT_OPT_DRY_RUN this initialises CUDA on opt->device and allocates the
 * device status word. *out receives the handle; the caller frees it with destroy.
 * Errors: ERR_INVALID (bad options or out == NULL), ERR_CUDA. */
int32_t trident_scm_create(const trident_scm_options* opt, trident_compile_hook hook, void* user,
                           trident_scm_t** out);

/* Appends one version (§3.5: versions are tried in creation order). The descriptor is
 * validated and copied; its kernel entry is resolved now, so the hit path does no
 * lookup (§3.3: the kernel entry is resolved when the specialisation is built). RoPE
 * versions build a frequency table for (theta, D) -- theta^(-2i/D) in fp64, split into two
 * fp32 -- shared by versions with equal (theta, D); the kernels form cos and sin of the
 * angle from it. Readers see the new table atomically (copy-on-write);
 * calls already running keep the table they loaded. May be called from a hook.
 * *out_index (may be NULL) receives the new version's index.
 * Errors: ERR_INVALID (descriptor), ERR_CAPACITY (table full), ERR_CUDA. */
int32_t trident_scm_register_spec(trident_scm_t* scm, const trident_spec_desc* desc,
                                  int32_t* out_index);

/* Ordered dispatch (§3.2, Algorithm 1). Validates args (ERR_INVALID, the hook is not
 * called), then tries versions 0..n-1 in order; the first whose guard holds is
 * selected, its launch preconditions are checked (output overlap, ERR_INVALID), its
 * kernel parameters are packed and it is launched on `stream` (a cudaStream_t; NULL is
 * the legacy default stream). Returns OK with *out_selected = index. If every guard
 * fails: calls the hook (MISS_HANDLED, *out_selected = the index the hook registered
 * or -1), or returns MISS with *out_selected = -1 when no hook ran. A failed launch
 * returns ERR_CUDA at once; no further version is tried (Algorithm 1, raise e).
 * out_selected may be NULL. */
int32_t trident_scm_invoke(trident_scm_t* scm, const trident_args* args, void* stream,
                           int32_t* out_selected);

/* Invokes args[0..n-1] in order with one call (one boundary crossing per decoder step;
 * §3.5: the hit path stays on the compiled side of a single entry call from the caller).
 * Each element behaves as trident_scm_invoke. Stops at the first element that returns
 * an error or MISS and returns that status; the elements after it get TRIDENT_NOT_RUN
 * in out_selected (n entries, may be NULL). Returns OK if all hit, else MISS_HANDLED
 * if some misses were handled. */
int32_t trident_scm_invoke_seq(trident_scm_t* scm, const trident_args* args, int32_t n,
                               void* stream, int32_t* out_selected);

/* A decoder step's layer-chain calls with as few launches as the data allows: a step
 * toward the mega-kernel systems that §5 of the paper discusses as related work (several
 * operators per device launch), while keeping the paper's per-call guarded selection; the
 * paper itself launches once per call. Same contract as trident_scm_invoke_seq -- statuses, out_selected,
 * hook, statistics -- with one difference in how hits run: the calls are taken in chunks
 * of up to 48 (TRIDENT_STEP_MAX); a chunk of two or more calls runs as ONE launch when
 *   - every call hits (Algorithm 1, per call, including its launch preconditions),
 *   - every selected version is a layer chain (LAYER_CHAIN or LAYER_CHAIN_QKNORM) with the
 *     same kernel (same dtype, H and q/k-norm choice; theta may differ), and
 *   - the calls are independent: no output byte of one call is a byte of any tensor of
 *     another call (exact for row-strided views with equal strides, conservative
 *     otherwise), so running them together equals running them in order.
 * Otherwise the chunk runs call by call exactly as invoke_seq (so a miss, the hook and
 * errors are reported at their position). Chunks run in order on `stream`. A fused chunk
 * counts one invoke and one hit per call, plus fused_launches and fused_calls in the
 * statistics; no host time is recorded for it. If its launch fails, the call returns
 * ERR_CUDA with the chunk's out_selected set to the versions it selected and the calls
 * after the chunk set to TRIDENT_NOT_RUN. Host cost of the independence test: one sort of
 * the chunk's tensor extents (about 20 per call).
 * Replay: a fused chunk's outcome depends on nothing but its argument bytes (selection reads
 * them and a table that only grows, so a call's first match cannot change; the byte rules
 * and the packed kernel parameters read only them and state fixed when the SCM and its
 * versions were created). The SCM therefore keeps the last few fused chunks whose
 * fingerprint it had seen before (4 entries, about 110 KB each, allocated on the first
 * store); a chunk whose argument bytes equal a kept one is relaunched from the stored
 * parameter block, with the same statuses, out_selected and statistics as the full path
 * (plus step_replays; guard_evals does not grow). A decode loop that passes the same
 * buffers every step takes this path from its third step on. Device data may change freely
 * between steps: only the argument bytes are compared. TRIDENT_OPT_NO_STEP_REPLAY turns it
 * off. Thread-safe: a thread that finds the cache in use by another takes the full path. */
#define TRIDENT_STEP_MAX 48
int32_t trident_scm_invoke_step(trident_scm_t* scm, const trident_args* args, int32_t n,
                                void* stream, int32_t* out_selected);

/* Appends a version that invoke_tree can select: desc as for register_spec, plus the
 * recipe that binds a call's argument tree to desc->op's slots (§3.3). The recipe is
 * validated (well-formed tree, every slot bound exactly once, bind codes legal for each
 * kind) and copied. Such versions are also seen by invoke (which ignores recipes); versions
 * without a recipe are skipped by invoke_tree. Errors: as register_spec. */
int32_t trident_scm_register_tree_spec(trident_scm_t* scm, const trident_spec_desc* desc,
                                       const trident_recipe* recipe, int32_t* out_index);

/* Ordered dispatch over structured arguments (§3.3, §3.5). Validates the tree (node kinds,
 * child ranges after their parent, size and depth limits, DLTensor dtypes and devices;
 * ERR_INVALID, the hook is not called). Then, for each version with a recipe in creation
 * order: the recipe's structure and guarded constants are checked against the tree (a
 * failure is that version's miss); the consumed leaves and bound scalars form the op's
 * argument tuple, which is validated (ERR_INVALID ends the call: the bound arguments are
 * malformed) and guarded as in invoke; the first version whose checks all hold is launched
 * as invoke does. A miss calls the tree hook if one is set (MISS_HANDLED) or returns MISS.
 * Results are written to the output tensors the tree names; nothing is returned. */
int32_t trident_scm_invoke_tree(trident_scm_t* scm, const trident_node* nodes, int32_t nargs,
                                int32_t nnodes, void* stream, int32_t* out_selected);

/* Installs (or with NULL removes) the compile hook of invoke_tree; same rules as the
 * invoke hook (§3.5: the caller's compile path runs only on a miss, never from inside a
 * hook). Errors: ERR_INVALID (scm NULL). */
int32_t trident_scm_set_tree_hook(trident_scm_t* scm, trident_tree_hook hook, void* user);

/* Selection only: validation plus Algorithm 1's guard loop, with no launch, no hook
 * and no statistics. Returns OK (*out_selected = index), MISS (-1) or ERR_INVALID.
 * Needs no GPU. */
int32_t trident_scm_select(const trident_scm_t* scm, const trident_args* args,
                           int32_t* out_selected);

/* Copies the counters into *out (calls, hits, misses, hook calls and failures, errors,
 * guard evaluations, fused launches, replayed calls). §4.1 measures a warm path: calls
 * that stay on the compiled hit path (§3.5: only a miss returns to the compile path),
 * timed on the host until the call returns and end to end until the device finishes;
 * these counters show which path each call took, and trident_scm_host_times gives the
 * host time of the hits. Each counter is read on its own, so counters that concurrent
 * invokers are updating may be a few calls apart. Errors: ERR_INVALID (scm or out NULL). */
int32_t trident_scm_stats(const trident_scm_t* scm, trident_scm_stats_t* out);

/* Copies per-version hit counts into out[0..cap-1]; *n (may be NULL) gets the count.
 * §3.5: versions are tried in creation order and later compatible calls use a newly
 * installed version; these counts show which version each hit selected (index order is
 * creation order). Errors: ERR_INVALID (scm NULL, cap < 0, or out NULL with cap > 0). */
int32_t trident_scm_spec_hits(const trident_scm_t* scm, uint64_t* out, int32_t cap, int32_t* n);

/* §4.1 and §2.3: host latency is the time until the call returns to its caller, read on
 * the warm path over many repeated calls (median and spread).
 * With TRIDENT_OPT_TIMING: copies the host nanoseconds of the most recent hits (entry
 * of invoke to return, launch included) into out[0..cap-1], oldest first; *n gets the
 * count. Samples are recorded per hit (and per launch of trident_launch_floor), so
 * concurrent invokers may interleave. Errors: ERR_INVALID (scm NULL, cap < 0, or out NULL
 * with cap > 0), ERR_STATE (TRIDENT_OPT_TIMING off). */
int32_t trident_scm_host_times(const trident_scm_t* scm, uint32_t* out, int32_t cap, int32_t* n);

/* Latency-floor probe (measurement, not part of the dispatch path; the paper has no such
 * probe). §2.3: on short kernels what remains on the warm path is host and launch cost,
 * and §4.1 reads end-to-end latency until the device finishes; this probe gives the part
 * of both that no dispatcher can remove, one launch. It launches n empty
 * kernels (one block of 32 threads; the kernel only takes part in programmatic dependent
 * launch) back to back on `stream`, with the SCM's launch configuration (its context, and
 * programmatic stream serialisation when TRIDENT_OPT_PDL is set) through the same driver
 * entry point as a hit. The time per launch is the single-launch floor against which
 * decode-size steps are reported. With TRIDENT_OPT_TIMING each launch's host nanoseconds
 * (the launch call alone: no guards, no packing) go to the host-time ring, the baseline
 * against which a hit's host time is read. Reads and writes no memory. Errors:
 * ERR_INVALID (scm NULL or n < 0), ERR_STATE (dry-run SCM), ERR_CUDA. */
int32_t trident_launch_floor(trident_scm_t* scm, void* stream, int32_t n);

/* Copy-floor probe (measurement, not part of the dispatch path; the paper has no such
 * probe). §4.1 reads end-to-end latency until the device finishes; for a memory-bound
 * launch that time is bounded below by moving its bytes, which this probe measures: n launches, back to back on
 * `stream` through the same launch code as a hit, of a kernel with a layer chain's traffic
 * and none of its arithmetic. Launch i reads read_bytes at src + (i % sets) * read_bytes and
 * writes write_bytes at dst + (i % sets) * write_bytes with a grid of `blocks` blocks of 256
 * threads: block b reads its even share of the 16-byte vectors and writes its even share,
 * every written vector the XOR of the vectors its thread read; with TRIDENT_OPT_PDL each
 * block first prefetches its read lines into L2 before its programmatic-launch wait, as the
 * layer chain's blocks do. Give it the bytes, block count and rotation of a chain launch and
 * the time per launch is what this GPU needs to move that traffic in that launch pattern: the
 * floor the chain kernel is read against. src and dst are device pointers (caller-owned,
 * 16-byte aligned, sets * read_bytes and sets * write_bytes long); the byte counts are
 * multiples of 16. Errors: ERR_INVALID (bad arguments), ERR_STATE (dry-run SCM), ERR_CUDA. */
int32_t trident_copy_floor(trident_scm_t* scm, void* stream, const void* src, void* dst, int64_t read_bytes,
                           int64_t write_bytes, int32_t blocks, int32_t sets, int32_t n);

/* Reads the device status word (TRIDENT_DEVERR_* bits) after synchronising `stream`;
 * clears it when clear != 0. §3.5: an execution error is a path of its own, never a miss
 * and never a reason to try another version; an error found inside a kernel (a position
 * outside the cache, a bounded wait that ran out) cannot return through the launch, so the
 * kernel sets its bit here and skips the faulty access, and the caller reads it after the
 * work has finished. Errors: ERR_INVALID (scm or out_bits NULL), ERR_STATE in dry-run mode,
 * ERR_CUDA. */
int32_t trident_scm_device_status(trident_scm_t* scm, void* stream, uint32_t* out_bits,
                                  int32_t clear);

/* RoPE + KV-cache append (ROPE_KV or QKNORM_ROPE_KV argument tuple, same slots and math)
 * that allocates nothing, for callers that cannot allocate device memory -- for example a
 * serving engine that has given all of HBM to its own pool, or code where a cudaMalloc
 * would synchronise the device. The paper has no counterpart: it is an addition of this
 * library. There is no SCM handle and no guard table: the call validates the tuple,
 * requires what the vector kernel needs (bf16 or fp16, D in {64, 128, 256}, 16-byte
 * aligned tensors, dense caches, tensors on the current device) and launches on `stream`.
 * Its scratch -- the status word and the RoPE frequency table -- lives in one static
 * device array of 256 + 1024 bytes that every GPU loading the library holds until exit;
 * a head size above 256 (more than 128 frequency pairs) is rejected with ERR_INVALID.
 * The first call on a device looks up the array's device address (cudaGetSymbolAddress),
 * so make that first call before any stream capture. Every call shares the array, which
 * keeps the last call's contents: each call first launches, on `stream`, a small kernel
 * that clears the status word and rewrites the table for the call's own (theta, D), so
 * nothing depends on what an earlier call left there. Calls that overlap on the GPU
 * (other streams, other host threads) race on the array. *out_status (may be NULL)
 * receives the status word (TRIDENT_DEVERR_* bits) by a cudaMemcpyAsync on `stream`
 * after the RoPE kernel; read it after synchronising the stream. Into page-locked host
 * memory that copy is asynchronous; into pageable memory it makes the host wait until the
 * kernel has finished. Errors: ERR_INVALID, ERR_CUDA. */
int32_t trident_rope_kv_noalloc(const trident_args* args, void* stream, uint32_t* out_status);

/* Frees the SCM, its tables and device memory. §3.4: the callable keeps the compiled
 * engine alive, so everything a version needs stays valid for as long as the callable
 * exists; here the handle is that callable, and it owns its versions, resolved kernels,
 * frequency tables and status word until this call ends its lifetime. The caller must
 * ensure no call on it is running and its kernels have finished. NULL is ignored. */
void trident_scm_destroy(trident_scm_t* scm);

/* Thread-local message of the last error returned on this thread ("" if none). §3.2 and
 * §3.4-3.5: an execution error ends dispatch and reaches the caller through the FFI's
 * error channel, distinct from a miss; the negative status says which kind of error and
 * this message says what failed. The buffer belongs to the calling thread and is
 * overwritten by that thread's next failing call. */
const char* trident_scm_last_error(void);

/* Static name of a status code (§3.4-3.5: a miss and an execution error are distinct
 * outcomes; the name says which). Unknown codes give "UNKNOWN". Never fails. */
const char* trident_status_name(int32_t status);

#ifdef __cplusplus
}
#endif
#endif /* TRIDENT_SCM_H */

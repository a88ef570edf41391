/*
 * fastcoder.h - C ABI of the GB300 retrieve-and-verify step of FastCoder
 * (arXiv 2502.17139): suffix-array draft retrieval from one or two token
 * datastores, weighted draft-tree construction, tree-masked verification
 * attention and greedy acceptance, plus the cache append that closes a
 * decoding step.
 *
 * Conventions for every call
 *   - Every pointer named d_* is DEVICE memory owned by the caller; the
 *     library never allocates, frees or retains it beyond the call.  Plain
 *     (non d_) pointers are host memory read during the call only.
 *   - Calls are asynchronous on the given stream (fc_stream = cudaStream_t;
 *     NULL is the legacy default stream) unless stated otherwise.  FC_OK
 *     means "arguments valid and work enqueued".  Errors that only the GPU
 *     can see (a token id >= vocab, a cache overflow, a bounded wait that ran
 *     out) are recorded in a device error word that fc_get_error() reads.
 *   - A host-detected error returns before anything is enqueued and leaves
 *     every output untouched.
 *   - Token ids are uint32 < vocab.  FC_PAD_TOKEN pads draft slots.
 *   - bf16 tensors are raw IEEE bfloat16 (2 bytes, little endian).
 *   - Outputs do not depend on the launch configuration (bit-exact
 *     determinism for integer outputs).
 */
#ifndef FASTCODER_H_
#define FASTCODER_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  FC_OK = 0,
  FC_ERR_INVALID_ARG = 1,  /* bad pointer, size, layout or value */
  FC_ERR_UNSUPPORTED = 2,  /* valid in principle, outside what the kernels support */
  FC_ERR_WORKSPACE = 3,    /* workspace pointer missing or smaller than required */
  FC_ERR_CAPACITY = 4,     /* a cache, context or path would overflow its capacity */
  FC_ERR_TIMEOUT = 5,      /* a bounded device-side wait ran out; the kernel returned */
  FC_ERR_CUDA = 6,         /* a CUDA runtime/driver call failed */
  FC_ERR_INTERNAL = 7,     /* an internal consistency check failed */
  FC_ERR_IO = 8            /* a datastore file could not be written or read, or failed its checks */
} fc_status;

typedef void* fc_stream; /* cudaStream_t */

#define FC_PAD_TOKEN 0xFFFFFFFFu
#define FC_MAX_NMAX 32        /* longest suffix length tried */
#define FC_MAX_TOPK 256       /* drafts kept per query and source */
#define FC_MAX_DRAFT_LEN 16   /* tokens per draft */
#define FC_MAX_OCC 4096       /* occurrences examined per query and source */
#define FC_MAX_SOURCES 4      /* datastores searched in one call */
#define FC_MAX_NODES 128      /* draft-tree nodes (root included) */
#define FC_LCP_CAP 255        /* longest-common-prefix values are stored capped here */

/* Self-test of failure detection (no counterpart in the paper): one CTA
 * waits on an mbarrier phase with the kernels' bounded wait.  arrive != 0
 * completes the phase first (FC_OK from fc_get_error); arrive == 0 leaves it
 * pending, so the wait gives up after limit_cycles (1..4e9 SM cycles; a poll
 * may add ~0.5 ms) and fc_get_error reports FC_ERR_TIMEOUT.  Nothing faults or
 * hangs and the context stays usable. */
fc_status fc_selftest_wait(int arrive, unsigned long long limit_cycles, fc_stream s);

/* Human-readable name of a status code (static storage). */
const char* fc_status_string(fc_status s);

/* Library version, e.g. "0.1.0". */
const char* fc_version(void);

/*
 * Waits for the stream, then returns and clears the device error word
 * (the most severe device-detected error since the last call, or FC_OK).
 * Synchronous.  The word is shared by every stream of the process: with
 * work on several streams, have s wait for them first (or synchronize the
 * device), or an error recorded later on another stream is missed by this
 * call and reported by the next.  The native step executor can give each
 * sub-batch a word of its own instead (fc_pipeline_part.err, read by
 * fc_pipeline_error), so that its errors are attributed to it exactly.
 */
fc_status fc_get_error(fc_stream s);

/* ------------------------------------------------------------------------
 * Datastore (Section IV-A, Eq. 1-2; Section III-A).  Every position of a
 * token corpus splits it into a context (the tokens before) and a
 * continuation (the tokens after); the suffix array over the corpus turns
 * "which contexts end with this suffix" into one contiguous SA range.
 * ------------------------------------------------------------------------ */
typedef struct {
  const uint32_t* tokens;  /* device, [n_tokens] token ids < vocab, 16-byte aligned
                              (fc_retrieve reads it as 16-byte vectors) */
  const uint32_t* sa;      /* device, [n_tokens] suffix array of tokens */
  const uint32_t* bucket;  /* device, [vocab + 1]: bucket[v] = first SA index whose
                              suffix starts with a token >= v; bucket[vocab] = n_tokens */
  const uint8_t* lcp;      /* device, [n_tokens]: lcp[j] = length of the longest common
                              prefix of the suffixes at sa[j-1] and sa[j], capped at
                              FC_LCP_CAP; lcp[0] = 0 */
  uint64_t n_tokens;       /* 1 <= n_tokens < 2^32 - 1 */
  uint32_t vocab;          /* 1 <= vocab < 2^31 */
  const uint32_t* keys;    /* device, optional (NULL: not used): [n_tokens][8] suffix
                              keys from fc_datastore_keys, 32-byte aligned */
} fc_datastore;

/*
 * Suffix keys: an index over the suffix array, not a step of the paper.
 * Entry j (8 uint32, 32 bytes) holds sa[j] and the suffix's tokens 1..7
 * (FC_PAD_TOKEN past the corpus end).  With keys set in the datastore view,
 * fc_retrieve's binary-search probes read one 32-byte entry (one DRAM
 * sector) where they would read the suffix array and then the corpus: a
 * probe touches the corpus only when the pattern's first eight tokens tie
 * with the suffix's.  Results are identical with and without keys.
 *   ds      a built datastore (tokens and sa are read)
 *   d_keys  [n_tokens][8] uint32 out, 32-byte aligned (32 bytes per token)
 * Asynchronous.  The caller then sets ds.keys = d_keys in its view.
 */
fc_status fc_datastore_keys(const fc_datastore* ds, uint32_t* d_keys, fc_stream s);

/* Workspace bytes fc_datastore_build needs for n_tokens tokens. */
size_t fc_datastore_build_workspace(uint64_t n_tokens, uint32_t vocab);

/*
 * Builds the suffix array and first-token bucket table of a token corpus
 * (the datastore organisation of Section IV-A, after REST).
 *   d_tokens [n_tokens] uint32 ids < vocab (checked; FC_ERR_INVALID_ARG if not)
 *   d_sa     [n_tokens] uint32 out: sa[j] = start of the j-th smallest suffix;
 *            a suffix that is a proper prefix of another sorts first
 *   d_bucket [vocab + 1] uint32 out (see fc_datastore.bucket)
 *   d_lcp    [n_tokens] uint8 out (see fc_datastore.lcp): adjacent suffixes'
 *            common prefix lengths, which let retrieval group equal
 *            continuations without reading them
 *   d_ws     workspace of at least fc_datastore_build_workspace() bytes
 *   out      host struct filled with the datastore view (may be NULL)
 * Synchronous: returns when the build is finished (it reads a group count
 * back after every doubling round).
 */
fc_status fc_datastore_build(const uint32_t* d_tokens, uint64_t n_tokens, uint32_t vocab,
                             uint32_t* d_sa, uint32_t* d_bucket, uint8_t* d_lcp, void* d_ws,
                             size_t ws_bytes, fc_stream s, fc_datastore* out);

/*
 * The same build for callers that cannot allocate device memory.  The paper
 * has no counterpart: this is a deployment variant of fc_datastore_build.
 * Some callers cannot call cudaMalloc, e.g. a serving process whose memory
 * manager reserves all free device memory for its KV cache up front, or a
 * plugin inside an application that owns every device allocation.  This
 * entry point allocates nothing: its scratch space is a fixed 30 MiB array
 * compiled into the library, which every GPU that loads the library holds
 * until the process exits.  The caller still passes the corpus, d_sa,
 * d_bucket and d_lcp.
 *   n_tokens must be <= FC_NOALLOC_MAX_TOKENS; larger corpora return
 *   FC_ERR_CAPACITY (use fc_datastore_build with a workspace instead).
 * Under CUDA's default lazy module loading the array is placed on a device
 * by the first datastore build made there (this call or
 * fc_datastore_build), so that first call needs 30 MiB of free device
 * memory: a caller that reserves all free memory makes one call (any small
 * corpus) before reserving it.  Later calls allocate nothing.  Every call
 * looks up the array's device address on the current device; the first
 * call on a device loads the library's module there, so make it before any
 * stream capture.  All calls share the array and find the last call's
 * contents in it: calls whose work overlaps on the GPU (other streams,
 * other host threads) race on it and must not be made.  Synchronous, like
 * fc_datastore_build.
 */
#define FC_NOALLOC_MAX_TOKENS 1048576ull
fc_status fc_datastore_build_noalloc(const uint32_t* d_tokens, uint64_t n_tokens, uint32_t vocab,
                                     uint32_t* d_sa, uint32_t* d_bucket, uint8_t* d_lcp,
                                     fc_stream s, fc_datastore* out);

/*
 * A built datastore on disk (the paper builds its datastores offline, once:
 * Section IV-A, Section V-C).  One file holds the corpus, the suffix array,
 * the bucket table and the LCP array, little endian, after a 64-byte header
 * (magic "FCDSTORE", version 1, vocab, n_tokens, payload bytes, and an FNV-1a
 * checksum over the payload's 64-bit words); the layout is spelled out in
 * datastore_io.cu.  on_host != 0: the arrays are host memory (no CUDA call is
 * made); otherwise device memory, moved through a 64 MiB pinned staging
 * buffer that the call allocates and frees (these two calls are the only ones
 * in the library that allocate, host memory only).  Synchronous.
 *
 * fc_datastore_save: writes ds to path (replacing the file).  FC_ERR_IO when
 *   the file cannot be written.
 * fc_datastore_file_info: n_tokens and vocab from a file's header, so the
 *   caller can size the buffers.  FC_ERR_IO for a missing or foreign file.
 * fc_datastore_load: reads a file into the caller's buffers: tokens and sa
 *   [n_tokens] uint32 (tokens 16-byte aligned), bucket [vocab + 1] uint32,
 *   lcp [n_tokens] uint8; n_capacity and vocab_capacity bound what the
 *   buffers hold (FC_ERR_CAPACITY beyond them).  FC_ERR_IO for a missing,
 *   foreign, truncated or overlong file or a checksum mismatch; the buffers
 *   may then hold part of the file.  On success `out` (may be NULL) views
 *   the loaded store.
 */
fc_status fc_datastore_save(const char* path, const fc_datastore* ds, int on_host, fc_stream s);
fc_status fc_datastore_file_info(const char* path, uint64_t* n_tokens, uint32_t* vocab);
fc_status fc_datastore_load(const char* path, uint32_t* tokens, uint32_t* sa, uint32_t* bucket, uint8_t* lcp,
                            uint64_t n_capacity, uint32_t vocab_capacity, int on_host, fc_stream s,
                            fc_datastore* out);

/*
 * The reversed corpus out[i] = tokens[n_tokens - 1 - i] (device buffers of
 * n_tokens uint32, not overlapping), from which fc_datastore_build makes the
 * reversed-corpus datastore that fc_retrieve_rev takes.  Asynchronous.
 */
fc_status fc_reverse_tokens(const uint32_t* d_tokens, uint64_t n_tokens, uint32_t* d_out, fc_stream s);

/* ------------------------------------------------------------------------
 * Retrieval (Section III-A; Section IV-C, Algorithm 1 par_search; Section
 * V-C: n_max = 16).
 * ------------------------------------------------------------------------ */
typedef struct {
  int32_t n_max;       /* longest suffix length tried, 1..FC_MAX_NMAX */
  int32_t n_min;       /* shortest suffix length tried, 1..n_max */
  int32_t top_k;       /* drafts kept, 1..FC_MAX_TOPK */
  int32_t draft_len;   /* tokens per draft, 1..FC_MAX_DRAFT_LEN */
  uint32_t max_occ;    /* occurrences examined, 1..FC_MAX_OCC */
} fc_retrieve_params;

/*
 * For every query b and every source s: the longest n in
 * [n_min, min(n_max, ctx_len[b])] whose last-n-token context suffix occurs
 * in the corpus immediately before a position p <= n_tokens - 1 (so a
 * continuation exists); the first max_occ occurrences in suffix-array order
 * (the lexicographically smallest windows); their continuations
 * T[p .. min(p + draft_len, n_tokens)) grouped by equality (length
 * included); and the top_k groups by count descending, then token ids
 * ascending (a prefix before its extensions).
 *
 *   sources     host array [n_sources] of datastore views (1..FC_MAX_SOURCES)
 *   d_ctx       [batch][ctx_stride] uint32 contexts; query b is
 *               d_ctx[b][0 .. ctx_len[b]) (ctx_len[b] in [0, ctx_stride])
 *   d_skip      optional [batch] int32: nonzero leaves query b's outputs
 *               untouched (they were served by a retrieval cache); may be NULL
 * Outputs (source-major, [n_sources][batch]...):
 *   d_drafts    [S][batch][top_k][draft_len] uint32, FC_PAD_TOKEN past a
 *               draft's end and in absent slots
 *   d_draft_len [S][batch][top_k] int32 (0 in absent slots)
 *   d_count     [S][batch][top_k] uint32 occurrence counts (0 in absent slots)
 *   d_n_drafts  [S][batch] int32 number of drafts found (<= top_k)
 *   d_match_len [S][batch] int32 the matched suffix length n (0: no match)
 * A context token >= vocab makes that query match nothing and records
 * FC_ERR_INVALID_ARG in the device error word.
 */
fc_status fc_retrieve(const fc_datastore* sources, int n_sources, const uint32_t* d_ctx,
                      int ctx_stride, const int32_t* d_ctx_len, int batch, const int32_t* d_skip,
                      fc_retrieve_params p, uint32_t* d_drafts, int32_t* d_draft_len,
                      uint32_t* d_count, int32_t* d_n_drafts, int32_t* d_match_len, fc_stream s);

/*
 * fc_retrieve without the top-k (the input of the all-occurrence trie,
 * fc_build_tree_all): every distinct continuation among the first max_occ
 * occurrences, in ascending token order (a prefix before its extensions),
 * with its count.  p.top_k is not used; the output arrays have p.max_occ
 * slots per query and source: d_drafts [S][batch][max_occ][draft_len],
 * d_draft_len and d_count [S][batch][max_occ], d_n_drafts and d_match_len
 * [S][batch].  Everything else as fc_retrieve.
 */
fc_status fc_retrieve_all(const fc_datastore* sources, int n_sources, const uint32_t* d_ctx,
                          int ctx_stride, const int32_t* d_ctx_len, int batch, const int32_t* d_skip,
                          fc_retrieve_params p, uint32_t* d_drafts, int32_t* d_draft_len,
                          uint32_t* d_count, int32_t* d_n_drafts, int32_t* d_match_len, fc_stream s);

/*
 * fc_retrieve with the longest match found through the reversed corpus
 * (a retrieval variant of Section III-A): the context suffixes of lengths
 * 1, 2, ... read backwards are prefixes of one another, so in the suffix
 * array of the reversed corpus their ranges are nested and one narrowing
 * search, one token longer per step, finds n*; the forward suffix array is
 * then searched for n* alone.  The outputs are exactly fc_retrieve's.
 *   rev_sources host array [n_sources]: rev_sources[s] is the datastore of
 *               sources[s]'s corpus reversed (fc_reverse_tokens, then
 *               fc_datastore_build); its lcp is not read and may be NULL.
 *               n_tokens and vocab must equal sources[s]'s
 *               (FC_ERR_INVALID_ARG otherwise); that the corpus really is
 *               the reverse is the caller's contract.
 * Every other argument, limit and output as fc_retrieve.
 */
fc_status fc_retrieve_rev(const fc_datastore* sources, const fc_datastore* rev_sources, int n_sources,
                          const uint32_t* d_ctx, int ctx_stride, const int32_t* d_ctx_len, int batch,
                          const int32_t* d_skip, fc_retrieve_params p, uint32_t* d_drafts,
                          int32_t* d_draft_len, uint32_t* d_count, int32_t* d_n_drafts,
                          int32_t* d_match_len, fc_stream s);

/* ------------------------------------------------------------------------
 * Context-keyed retrieval cache (workload support for the step loop;
 * Section IV-B motivates caching retrieval results, this cache replays a
 * query's earlier result when its last n_max context tokens repeat).
 * The table lives in caller-owned device memory.
 * ------------------------------------------------------------------------ */
size_t fc_rcache_bytes(int capacity, int n_sources, fc_retrieve_params p);

/* Clears a table of `capacity` entries (a power of two, 1..2^24). */
fc_status fc_rcache_init(void* d_table, size_t bytes, int capacity, int n_sources,
                         fc_retrieve_params p, fc_stream s);

/*
 * For each query b with d_want_hit[b] != 0 whose key (its last
 * min(n_max, ctx_len[b]) tokens) is in the table, copies the stored
 * retrieval outputs into the output arrays (same layout as fc_retrieve) and
 * sets d_skip[b] = 1; otherwise sets d_skip[b] = 0.  d_want_hit may be NULL
 * (every query may hit).
 */
fc_status fc_rcache_lookup(const void* d_table, int capacity, int n_sources, fc_retrieve_params p,
                           const uint32_t* d_ctx, int ctx_stride, const int32_t* d_ctx_len,
                           int batch, const int32_t* d_want_hit, int32_t* d_skip,
                           uint32_t* d_drafts, int32_t* d_draft_len, uint32_t* d_count,
                           int32_t* d_n_drafts, int32_t* d_match_len, fc_stream s);

/*
 * fc_rcache_lookup and then fc_retrieve on the queries it did not serve, in
 * one launch: each (query, source) CTA first looks the query's key up and,
 * when served, copies its source's stored result; the others retrieve.  The
 * outputs and d_skip are exactly those of the two calls (a served query
 * records no token error, as there).  Arguments as the two calls; d_skip
 * [batch] is written (1 = served).
 */
fc_status fc_retrieve_cached(const fc_datastore* sources, int n_sources, const uint32_t* d_ctx,
                             int ctx_stride, const int32_t* d_ctx_len, int batch, const void* d_table,
                             int capacity, const int32_t* d_want_hit, int32_t* d_skip,
                             fc_retrieve_params p, uint32_t* d_drafts, int32_t* d_draft_len,
                             uint32_t* d_count, int32_t* d_n_drafts, int32_t* d_match_len, fc_stream s);

/*
 * Stores the retrieval outputs of every query with d_skip[b] == 0 under its
 * key (replacing an equal key).  A full table records FC_ERR_CAPACITY.
 */
fc_status fc_rcache_insert(void* d_table, int capacity, int n_sources, fc_retrieve_params p,
                           const uint32_t* d_ctx, int ctx_stride, const int32_t* d_ctx_len,
                           int batch, const int32_t* d_skip, const uint32_t* d_drafts,
                           const int32_t* d_draft_len, const uint32_t* d_count,
                           const int32_t* d_n_drafts, const int32_t* d_match_len, fc_stream s);

/* ------------------------------------------------------------------------
 * CACHE and missing table (Section IV-B; Section IV-C, Algorithm 1;
 * Section V-C: l = 50, the model's output stored in pieces of 20 tokens).
 *
 * Every sequence b of a batch owns a CACHE: a store of token sequences, each
 * either a verified retrieval (the last ctx_keep context tokens before a step
 * followed by the draft tokens that step accepted) or a complete piece of
 * `chunk` tokens of the model's output (the tokens appended to the context
 * after the prompt).  Once it holds min_size sequences or more, a CACHE is
 * searched before the datastore, with fc_retrieve's definition applied to
 * the stored sequences: a match lies inside one stored sequence and a
 * continuation stops at the end of its sequence.
 *
 * The missing table M (one per batch) holds the n_min-token context
 * suffixes for which every datastore source returned nothing.  A match of
 * length n implies matches of all shorter lengths at the same position, so
 * for a static datastore this key decides exactly whether retrieval can
 * return anything.  A context that ends with a key in M skips the datastore.
 *
 * Per step: fc_cache_search -> fc_retrieve (d_skip = the state array) ->
 * fc_missing_insert -> tree, verification, acceptance, fc_kv_append ->
 * fc_cache_update.
 *
 * CACHE layout (caller-owned device memory):
 *   d_words [batch][capacity] uint32: the stored sequences back to back,
 *           each followed by FC_SEP_TOKEN (a sequence of L tokens costs L+1
 *           words; one that does not fit is dropped and counted);
 *   d_meta  [batch][4] int32: words used, sequences stored, output mark (the
 *           context length where the next output piece starts), sequences
 *           dropped for lack of room.
 * M layout: uint32 words [0] keys stored, [1] keys dropped, [2..3] zero, then
 * `capacity` slots of 1 + key_len words (a nonzero tag, then the key).  M
 * holds at most capacity / 2 keys.
 * ------------------------------------------------------------------------ */
#define FC_SEP_TOKEN 0xFFFFFFFEu
#define FC_CACHE_MAX_WORDS 16384
#define FC_SERVE_DATASTORE 0 /* search the datastore sources */
#define FC_SERVE_CACHE 1     /* the CACHE returned drafts */
#define FC_SKIP_MISSING 2    /* the context's key is in M: no retrieval */

typedef struct {
  uint32_t* d_words;  /* [batch][capacity] */
  int32_t* d_meta;    /* [batch][4] */
  int32_t capacity;   /* words per sequence: a multiple of 4 in 16..FC_CACHE_MAX_WORDS */
  int32_t min_size;   /* l: stored sequences needed before a search, >= 0 */
  int32_t chunk;      /* output piece length, >= 1 */
  int32_t ctx_keep;   /* context tokens stored before a verified draft, 0..FC_MAX_NMAX */
} fc_cache;

/* Empties every CACHE; the output mark starts at d_prompt_len[b]. */
fc_status fc_cache_init(const fc_cache* cache, int batch, const int32_t* d_prompt_len, fc_stream s);

/* Bytes of a missing table with `capacity` slots (a power of two, 2..2^24)
 * and keys of key_len tokens (1..FC_MAX_NMAX); 0 for bad arguments. */
size_t fc_missing_bytes(int capacity, int key_len);

/* Empties a missing table. */
fc_status fc_missing_init(void* d_table, size_t bytes, int capacity, int key_len, fc_stream s);

/*
 * Algorithm 1 up to the datastore search.  The result arrays have the
 * fc_retrieve layout with n_sources + 1 slots ([n_sources + 1][batch]...):
 * slot n_sources receives the CACHE's result (empty while the CACHE holds
 * fewer than min_size sequences), and for every query not sent to the
 * datastore, slots 0..n_sources-1 are cleared.  d_state[b] gets
 * FC_SERVE_CACHE when the CACHE returned drafts, else FC_SKIP_MISSING when
 * the context's last p.n_min tokens are in M, else FC_SERVE_DATASTORE; pass
 * it to fc_retrieve as d_skip.  d_missing may be NULL (no table); its keys
 * are p.n_min tokens long.  Limits as fc_retrieve.
 */
fc_status fc_cache_search(const fc_cache* cache, const void* d_missing, int missing_capacity,
                          const uint32_t* d_ctx, int ctx_stride, const int32_t* d_ctx_len, int batch,
                          fc_retrieve_params p, int n_sources, uint32_t* d_drafts, int32_t* d_draft_len,
                          uint32_t* d_count, int32_t* d_n_drafts, int32_t* d_match_len, int32_t* d_state,
                          fc_stream s);

/*
 * Adds to M the key (last key_len context tokens) of every query with
 * d_state[b] == FC_SERVE_DATASTORE, ctx_len[b] >= key_len and no draft in
 * any of the n_sources datastore slots of d_n_drafts ([>= n_sources][batch],
 * fc_retrieve's output).  Keys new to M are admitted in query order while M
 * holds fewer than capacity / 2 keys; the others are counted as dropped.
 */
fc_status fc_missing_insert(void* d_missing, int missing_capacity, int key_len, const uint32_t* d_ctx,
                            int ctx_stride, const int32_t* d_ctx_len, int batch, const int32_t* d_state,
                            const int32_t* d_n_drafts, int n_sources, fc_stream s);

/*
 * The CACHE update after verification.  For a query whose context grew by
 * acc_len + 1 tokens this step (d_ctx_len_new = d_ctx_len_old + acc_len + 1)
 * and acc_len >= 1, stores ctx[old - min(ctx_keep, old) .. old + acc_len)
 * (the verified retrieval: context suffix, then the accepted draft tokens).
 * Then, while d_ctx_len_new - mark >= chunk, stores ctx[mark .. mark + chunk)
 * and advances the mark.  A token >= FC_SEP_TOKEN in a sequence to store
 * records FC_ERR_INVALID_ARG and that sequence is skipped.
 */
fc_status fc_cache_update(const fc_cache* cache, const uint32_t* d_ctx, int ctx_stride,
                          const int32_t* d_ctx_len_old, const int32_t* d_ctx_len_new, const int32_t* d_acc_len,
                          int batch, fc_stream s);

/* ------------------------------------------------------------------------
 * Draft tree (Section IV-D: Eq. 3 node weight alpha*t_r + beta*t_c, the
 * top-weighted trie nodes as the draft; Eq. 4 tree mask; position ids by
 * depth; Section V-C: alpha = beta = 1, at most 64 draft tokens).
 * ------------------------------------------------------------------------ */
/*
 * Merges the drafts of n_sources sources (the fc_retrieve output layout)
 * into one trie per query rooted at d_root_tok[b] (the last context token,
 * whose K/V is not yet cached).  A draft u weighs
 * w(u) = sum_s src_weight[s] * count_s(u); a node weighs the sum of w over
 * the drafts through it.  The root and the node_budget - 1 heaviest other
 * nodes (ties: shallower first, then smaller token path) are kept and
 * emitted in depth-first preorder with children in ascending token order.
 *   src_weight  host [n_sources] uint32 (alpha, beta), each <= 65535
 *   node_budget 1..n_pad, n_pad in {64, 128}
 * Outputs, [batch][n_pad] unless noted; rows >= n_nodes[b] are padding
 * (tok = FC_PAD_TOKEN, parent = depth = pos = -1, mask = 0):
 *   d_tok, d_parent (parent[0] = -1, parent[i] < i), d_depth (root 0),
 *   d_pos (= kv_len[b] + depth), d_mask [batch][n_pad][n_pad/64] uint64 with
 *   bit j of row i set iff node j is an ancestor of node i or i itself,
 *   d_n_nodes [batch].
 * Limits: n_sources * top_k <= 512, draft_len <= FC_MAX_DRAFT_LEN.
 */
fc_status fc_build_tree(int n_sources, const uint32_t* d_drafts, const int32_t* d_draft_len,
                        const uint32_t* d_count, const int32_t* d_n_drafts,
                        const uint32_t* src_weight, int top_k, int draft_len,
                        const uint32_t* d_root_tok, const int32_t* d_kv_len, int batch,
                        int node_budget, int n_pad, uint32_t* d_tok, int32_t* d_parent,
                        int32_t* d_depth, int32_t* d_pos, uint64_t* d_mask, int32_t* d_n_nodes,
                        fc_stream s);

/*
 * The all-occurrence trie (Section III-A, Eq. 3 over every retrieved
 * continuation instead of the top-k): fc_build_tree's tree over the
 * drafts that fc_retrieve_all writes, every distinct continuation of each
 * source with its count.  Each source's valid drafts (the first
 * n_drafts[s][b] slots with 1 <= draft_len <= draft_len) must be in strictly
 * ascending token order (a prefix before its extensions), as
 * fc_retrieve_all writes them; a query that breaks this records
 * FC_ERR_INVALID_ARG and gets a root-only tree.
 *   d_drafts    [n_sources][batch][slots][draft_len] (the fc_retrieve_all
 *               layout, slots = its max_occ); d_draft_len, d_count
 *               [n_sources][batch][slots]; d_n_drafts [n_sources][batch]
 *   d_ws        device workspace, 256-byte aligned, of at least
 *               fc_build_tree_all_workspace(n_sources, slots, draft_len, batch)
 *               bytes (FC_ERR_WORKSPACE otherwise)
 * Weights, budget, tie-breaks and outputs as fc_build_tree.  Counts above
 * 2^17 are clamped (FC_ERR_INVALID_ARG recorded).
 * Limits: n_sources * slots <= 8192, draft_len <= FC_MAX_DRAFT_LEN.
 */
size_t fc_build_tree_all_workspace(int n_sources, int slots, int draft_len, int batch);
fc_status fc_build_tree_all(int n_sources, const uint32_t* d_drafts, const int32_t* d_draft_len,
                            const uint32_t* d_count, const int32_t* d_n_drafts, const uint32_t* src_weight,
                            int slots, int draft_len, const uint32_t* d_root_tok, const int32_t* d_kv_len,
                            int batch, int node_budget, int n_pad, void* d_ws, size_t ws_bytes,
                            uint32_t* d_tok, int32_t* d_parent, int32_t* d_depth, int32_t* d_pos,
                            uint64_t* d_mask, int32_t* d_n_nodes, fc_stream s);

/*
 * Eq. 4 mask, depths and position ids of trees given by parent pointers in
 * the layout above (parent[0] = -1, 0 <= parent[i] < i for 0 < i < n_nodes).
 * A malformed parent records FC_ERR_INVALID_ARG and zeroes that tree's mask.
 */
fc_status fc_tree_mask(const int32_t* d_parent, const int32_t* d_n_nodes, const int32_t* d_kv_len,
                       int batch, int n_pad, int32_t* d_depth, int32_t* d_pos, uint64_t* d_mask,
                       fc_stream s);

/* ------------------------------------------------------------------------
 * Verification attention (Section IV-D, Eq. 4): every tree node attends to
 * the whole KV cache and to its tree ancestors (and itself), one forward for
 * all drafts.
 * ------------------------------------------------------------------------ */
/*
 * out[b][i][h] = sum_j softmax_j(scale * q[b][i][h] . k_j) v_j over the keys
 * j = every cached key of kv head g = h / (H / Hkv) at positions
 * [0, kv_len[b]) and every tree key j with bit j of mask[b][i] set.
 * Rows i >= n_nodes[b] are written as zeros.  Q and K arrive already
 * position-encoded (the caller applies the depth-based position ids).
 *   d_q       bf16 [batch][n_pad][H][D]
 *   d_k_cache, d_v_cache  bf16 [batch][Hkv][kv_cap][D]
 *   d_kv_len  [batch] int32, 0 <= kv_len <= kv_cap (checked on the device)
 *   d_k_tree, d_v_tree    bf16 [batch][Hkv][n_pad][D] (the tree tokens' K/V)
 *   d_mask    [batch][n_pad][n_pad/64] uint64 (fc_build_tree layout)
 *   d_n_nodes [batch] int32 in [1, n_pad]
 *   d_out     bf16 [batch][n_pad][H][D]
 *   d_ws, ws_bytes  optional device workspace (may be NULL / 0).  With
 *             fc_tree_attn_workspace() bytes the call may split each row
 *             chunk's keys over up to 4 CTAs (so that the grid fills the GPU
 *             in whole waves) and merge their partial softmax sums; with less
 *             it uses fewer parts.  Owned by the caller, no initial contents
 *             needed (the call clears its counters on the stream first).
 *             Concurrent calls on different streams need separate workspaces.
 * Supported: D = 128, n_pad in {64, 128}, H % Hkv == 0, H / Hkv <= 16,
 * all device pointers 16-byte aligned.  Arithmetic: bf16 tensor-core
 * products with fp32 accumulation and an fp32 online softmax; the split
 * merge is fp32.  Results agree to rounding for every workspace size.
 */
fc_status fc_tree_attn(const void* d_q, const void* d_k_cache, const void* d_v_cache, int kv_cap,
                       const int32_t* d_kv_len, const void* d_k_tree, const void* d_v_tree,
                       const uint64_t* d_mask, const int32_t* d_n_nodes, int batch, int n_pad,
                       int H, int Hkv, int D, float scale, void* d_out, void* d_ws,
                       size_t ws_bytes, fc_stream s);

/* Workspace bytes that let fc_tree_attn use its largest key split for this
 * shape (0 for an unsupported shape).  Not part of the paper's method: a
 * scheduling aid for filling the GPU. */
size_t fc_tree_attn_workspace(int batch, int n_pad, int H, int Hkv);

/* 1 if fc_tree_attn serves this shape with its streaming kernel on the
 * current device, else 0 (also for an unsupported shape).  The streaming
 * kernel takes launches whose groups fit one 128-row tile (H / Hkv * n_pad
 * <= 128) and whose caches are short, with several groups per SM: each CTA
 * serves groups in turn and overlaps one group's epilogue with the next one's
 * query staging and first blocks.  Results equal the per-group kernel's.
 * Host-only, launches nothing. */
int fc_tree_attn_streamed(int batch, int n_pad, int H, int Hkv, int kv_cap);

/* How many parts fc_tree_attn splits each row chunk's keys into for this
 * shape and workspace size on the current device (1 = no split; 0 for an
 * unsupported shape).  Host-only, launches nothing. */
int fc_tree_attn_parts(int batch, int n_pad, int H, int Hkv, int kv_cap, size_t ws_bytes);

/* ------------------------------------------------------------------------
 * Rotary position embedding by node position (Section IV-D: the tree's tokens
 * take adjusted position indices, kv_len + depth, which fc_build_tree writes
 * to d_pos).  RoPE (Su et al., RoFormer) with the rotate-half pairing of the
 * LLaMA family: dimension i pairs with i + D/2 and turns by
 * pos * base^(-2i/D).  Angles in fp32, reduced modulo 2 pi before the
 * sine and cosine; results rounded to bf16.  A negative position (a padding
 * row of a tree) leaves its row unchanged.
 * ------------------------------------------------------------------------ */
/*
 * Rotates bf16 rows: layout 0 = node-major [batch][n_pad][heads][D] (queries),
 * layout 1 = head-major [batch][heads][n_pad][D] (tree keys); row (b, i, h)
 * turns by d_pos[b][i].  d_out may equal d_in.  D a multiple of 16 up to
 * 1024; pointers 16-byte aligned; base > 0.
 */
fc_status fc_rope(const void* d_in, void* d_out, int batch, int n_pad, int heads, int D, int layout,
                  const int32_t* d_pos, float base, fc_stream s);

/*
 * fc_tree_attn with unrotated queries: the query of node i is rotated by
 * d_pos[b][i] inside the kernel, while its tile is staged.  d_k_tree must
 * hold the tree keys already rotated (fc_rope, layout 1, the same d_pos and
 * base); the cached keys are the rotated keys of earlier steps.  Limits and
 * workspace as fc_tree_attn.
 */
fc_status fc_tree_attn_rope(const void* d_q, const void* d_k_cache, const void* d_v_cache, int kv_cap,
                            const int32_t* d_kv_len, const void* d_k_tree, const void* d_v_tree,
                            const uint64_t* d_mask, const int32_t* d_n_nodes, int batch, int n_pad,
                            int H, int Hkv, int D, float scale, const int32_t* d_pos, float rope_base,
                            void* d_out, void* d_ws, size_t ws_bytes, fc_stream s);

/* ------------------------------------------------------------------------
 * The decoder around the tree attention (Section IV-D: the target model
 * verifies every draft in one forward).  Building blocks of a LLaMA-family
 * decoder like the paper's models: embedding, residual add + RMSNorm, the
 * SiLU-gated MLP activation, the head-major layout of the tree's keys
 * (rotated) and values, and plain GEMMs.  bf16 tensors, row-major, 16-byte
 * aligned; fp32 arithmetic inside.
 * ------------------------------------------------------------------------ */
/* Workspace bytes fc_gemm_bf16 uses: 0 (the arguments stay for callers that
 * pass a buffer; it is not read). */
size_t fc_gemm_workspace(void);

/* C[M][N] = A[M][K] B[K][N], row-major bf16 (A the activations, B the weights
 * as stored, [K][N]), fp32 accumulation, C rounded to bf16.  The library's
 * own tcgen05 kernel: tiles of 128 x 256, TMA-fed, accumulators in tensor
 * memory, persistent over the GPU's SMs.  N and K multiples of 8 (else
 * FC_ERR_UNSUPPORTED); pointers 16-byte aligned.  Asynchronous; a bounded
 * wait that runs out sets FC_ERR_TIMEOUT in the device error word. */
fc_status fc_gemm_bf16(const void* d_a, const void* d_b, void* d_c, int M, int N, int K, void* d_ws,
                       size_t ws_bytes, fc_stream s);

/* The decoder's K/V projection with its next step folded into the GEMM's
 * epilogue: kv = A[M][K] Wkv[K][2 Hkv D] (Hkv key heads, then Hkv value heads
 * of D = 128 columns), rows (sequence b, node i) = b * n_pad + i, M = batch *
 * n_pad.  From the fp32 accumulators the key heads are rotated by d_pos[b][i]
 * (RoPE, rotate-half pairing, as fc_rope; a negative position leaves the row
 * unrotated), and both are written head-major and rounded once to bf16:
 * d_k_rot and d_v_heads [batch][Hkv][n_pad][D], the layout fc_tree_attn and
 * fc_kv_append read.  D != 128 or K % 8 gives FC_ERR_UNSUPPORTED. */
fc_status fc_gemm_kv_heads(const void* d_a, const void* d_wkv, int M, int K, int Hkv, int D, int batch, int n_pad,
                           const int32_t* d_pos, float rope_base, void* d_k_rot, void* d_v_heads, fc_stream s);

/* The gate/up projection with the SiLU-gated product folded into the GEMM's
 * epilogue: act[M][inter] = silu(A Wg) * (A Wu), fp32 inside, rounded once
 * to bf16.  d_wgu holds Wg and Wu interleaved in 128-column blocks, as
 * fc_interleave_gate_up writes them.  inter % 128 or K % 8 gives
 * FC_ERR_UNSUPPORTED. */
fc_status fc_gemm_silu_mul(const void* d_a, const void* d_wgu, int M, int K, int inter, void* d_act, fc_stream s);

/* Weight preparation for fc_gemm_silu_mul (once, at load): d_wgu [K][2 inter]
 * (the gate columns, then the up columns) -> d_out [K][2 inter] with block t
 * of 256 columns = gate columns 128t .. 128t+127, then up columns 128t ..
 * 128t+127.  Buffers must not overlap. */
fc_status fc_interleave_gate_up(const void* d_wgu, void* d_out, int K, int inter, fc_stream s);

/* out[t][:] = table[tok[t]][:]; an id >= vocab (tree padding) gives zeros.
 * hidden a multiple of 8. */
fc_status fc_embed(const uint32_t* d_tok, int n, const void* d_table, int vocab, int hidden, void* d_out,
                   fc_stream s);

/* Per row: if d_r, x += r (in place, rounded to bf16: the residual stream);
 * then out = x / sqrt(mean(x^2) + eps) * w.  dim a multiple of 8. */
fc_status fc_add_rmsnorm(void* d_x, const void* d_r, const void* d_w, void* d_out, int rows, int dim,
                         float eps, fc_stream s);

/* out[r][j] = silu(gu[r][j]) * gu[r][inter + j], silu(z) = z / (1 + e^-z):
 * gu holds the gate columns, then the up columns. */
fc_status fc_silu_mul(const void* d_gu, void* d_out, int rows, int inter, fc_stream s);

/* Node-major projection rows in[(b * n_pad + i) * in_stride + h * D + d]
 * (elements) to head-major out[b][h][i][d], rotated as fc_rope by
 * d_pos[b][i] when base > 0, copied when base <= 0 (the values). */
fc_status fc_rope_heads(const void* d_in, int in_stride, void* d_out, int batch, int n_pad, int heads, int D,
                        const int32_t* d_pos, float base, fc_stream s);

/* ------------------------------------------------------------------------
 * Acceptance (Section IV-D: every correct token from the start is accepted,
 * everything after the first error rejected; Eq. 7 counts tokens per step).
 * ------------------------------------------------------------------------ */
/*
 * Walks each tree from the root: at node cur, if some child carries the
 * target model's prediction d_argmax[b][cur], move to it; otherwise stop.
 *   d_acc_len [batch] int32 draft tokens accepted
 *   d_path    [batch][path_cap] int32 node ids path[0] = 0 .. path[acc_len],
 *             -1 after
 *   d_bonus   [batch] uint32 the prediction at the last accepted node
 * A path longer than path_cap records FC_ERR_CAPACITY (it is cut there).
 */
fc_status fc_accept(const uint32_t* d_tok, const int32_t* d_parent, const int32_t* d_n_nodes,
                    const uint32_t* d_argmax, int batch, int n_pad, int32_t* d_acc_len,
                    int32_t* d_path, int path_cap, uint32_t* d_bonus, fc_stream s);

/*
 * Greedy verification straight from the target model's logits (Section IV-D:
 * each draft token is checked against the model's most likely next token):
 * the argmax of every tree node's logits row, then the walk of fc_accept.
 *   d_logits  bf16 [batch][n_pad][vocab]; rows i >= n_nodes[b] are not read;
 *             2-byte aligned (rows need not be 16-byte aligned)
 *   d_argmax  [batch][n_pad] uint32 out: the prediction at every node (0 for
 *             rows >= n_nodes)
 *   the other arguments and outputs as fc_accept
 * Ties go to the smallest index; a NaN counts as larger than every number and
 * the first NaN wins (the convention of torch.argmax).  Each valid row is read
 * once with 16-byte loads (HBM-bound).  Two kernels on `s`.
 */
fc_status fc_argmax_accept(const void* d_logits, int vocab, const uint32_t* d_tok,
                           const int32_t* d_parent, const int32_t* d_n_nodes, int batch,
                           int n_pad, uint32_t* d_argmax, int32_t* d_acc_len, int32_t* d_path,
                           int path_cap, uint32_t* d_bonus, fc_stream s);

/*
 * Closes a decoding step: copies the K/V rows of the accepted path (root
 * included) to cache rows kv_len_in[b] .. kv_len_in[b] + acc_len[b],
 * writes kv_len_out = kv_len_in + acc_len + 1, appends the accepted draft
 * tokens and the bonus token to the context (ctx_len_out likewise) and
 * writes the bonus token to d_root_out (the next step's root).
 * In and out length arrays must not alias.  An overflow of kv_cap or
 * ctx_stride records FC_ERR_CAPACITY and leaves that sequence unchanged
 * (its out lengths equal its in lengths).
 */
fc_status fc_kv_append(const int32_t* d_path, const int32_t* d_acc_len, const uint32_t* d_bonus,
                       const uint32_t* d_tok, const void* d_k_tree, const void* d_v_tree,
                       int batch, int n_pad, int Hkv, int D, int path_cap, void* d_k_cache,
                       void* d_v_cache, int kv_cap, const int32_t* d_kv_len_in,
                       int32_t* d_kv_len_out, uint32_t* d_ctx, int ctx_stride,
                       const int32_t* d_ctx_len_in, int32_t* d_ctx_len_out,
                       uint32_t* d_root_out, fc_stream s);

/* ------------------------------------------------------------------------
 * Synthetic target model (workload scaffolding, not part of the method;
 * the paper's target model is an LLM whose greedy predictions drive
 * acceptance).  Along the tree's first branch the model agrees with the
 * tree for d_plen[b] steps; every other prediction is d_rtok[b][i] moved up
 * by one (mod vocab) while it equals the token of a child of node i, at most
 * n_pad times (if the children cover the whole vocabulary the last candidate
 * stands).
 * ------------------------------------------------------------------------ */
fc_status fc_synth_argmax(const uint32_t* d_tok, const int32_t* d_parent, const int32_t* d_n_nodes,
                          int batch, int n_pad, const int32_t* d_plen, const uint32_t* d_rtok,
                          uint32_t vocab, uint32_t* d_argmax, fc_stream s);

/* ------------------------------------------------------------------------
 * Native step executor (the decoding step of Section IV-C and IV-D over
 * sub-batches: replay-cache lookup -> fc_retrieve -> insert (or Algorithm
 * 1's CACHE search -> fc_retrieve -> missing-table insert) ->
 * fc_build_tree -> [fc_rope] -> fc_tree_attn[_rope] -> fc_synth_argmax ->
 * fc_accept -> fc_kv_append [-> fc_cache_update]).  One call enqueues the whole step of every
 * sub-batch; each sub-batch runs on two streams the executor owns, a
 * high-priority one for its latency-bound chain and a low-priority one for
 * its attention, so sub-batches overlap.  The executor owns no device
 * memory: all buffers below belong to the caller and must outlive it.
 * ------------------------------------------------------------------------ */
typedef struct {
  int32_t batch;            /* sequences in this sub-batch (>= 1) */
  int32_t first;            /* index of its first sequence in the batch-wide step inputs */
  uint32_t* ctx;            /* [batch][ctx_stride] contexts, appended to in place */
  int32_t ctx_stride;
  int32_t* ctx_len[2];      /* [batch] each; a step of phase c reads [c] and writes [1 - c] */
  int32_t* kv_len[2];       /* [batch] each; as ctx_len */
  uint32_t* root;           /* [batch] the next tree's root token, rewritten by each step */
  void* rcache;             /* fc_rcache_init'ed table, or NULL (no replay cache) */
  int32_t rcache_capacity;
  int32_t* skip;            /* [batch] scratch: queries the replay cache served */
  /* retrieval outputs, fc_retrieve's layout with top_k slots */
  uint32_t* drafts;
  int32_t* draft_len;
  uint32_t* count;
  int32_t* n_drafts;
  int32_t* match_len;
  /* tree outputs, fc_build_tree's layout */
  uint32_t* tok;
  int32_t* parent;
  int32_t* depth;
  int32_t* pos;
  uint64_t* mask;
  int32_t* n_nodes;
  void* k_cache;            /* bf16 [batch][Hkv][kv_cap][D]: this sub-batch's rows */
  void* v_cache;
  void* k_tree_rot;         /* bf16 [batch][Hkv][n_pad][D] rotated tree keys (RoPE only, else NULL) */
  void* attn_out;           /* bf16 [batch][n_pad][H][D] */
  void* attn_ws;            /* fc_tree_attn workspace of this sub-batch (NULL: no key split) */
  size_t attn_ws_bytes;
  uint32_t* argmax;         /* [batch][n_pad] */
  int32_t* acc_len;         /* [batch] */
  int32_t* path;            /* [batch][path_cap] */
  uint32_t* bonus;          /* [batch] */
  uint32_t* err;            /* this sub-batch's device error word (4 bytes, zeroed by the
                               caller; fc_pipeline_error reads it), or NULL: its kernels
                               then record errors in the library-wide words of fc_get_error */
  /* Algorithm 1 (Section IV-B/C) in place of the replay cache (rcache must then be NULL):
   * fc_cache_search -> fc_retrieve of the queries it leaves to the datastore ->
   * fc_missing_insert, and fc_cache_update after the append.  The retrieval outputs
   * above then hold n_sources + 1 slots, the CACHE's last, and `skip` holds the
   * search's per-query state. */
  fc_cache seq_cache;       /* this sub-batch's CACHE (fc_cache_init'ed); d_words NULL: none */
  void* missing;            /* this sub-batch's missing table M (fc_missing_init'ed with key
                               length n_min), or NULL: no M */
  int32_t missing_capacity;
} fc_pipeline_part;

typedef struct {
  const fc_datastore* sources;  /* host [n_sources], copied at creation */
  int32_t n_sources;
  fc_retrieve_params p;
  const uint32_t* src_weight;   /* host [n_sources] tree weights (Eq. 3), copied */
  int32_t node_budget, n_pad, H, Hkv, D, kv_cap, path_cap;
  uint32_t vocab;               /* the synthetic target model's vocabulary */
  float scale;                  /* attention scale (> 0) */
  float rope_base;              /* 0: q and tree keys arrive rotated; > 0: RoPE base */
  int32_t n_parts;
  const fc_pipeline_part* parts;  /* host [n_parts], copied */
  uint32_t cache_weight;        /* tree weight of the CACHE slot (parts with a CACHE) */
} fc_pipeline_desc;

typedef struct fc_pipeline fc_pipeline;

/* Checks the description (FC_ERR_INVALID_ARG: a missing buffer, a
 * non-positive size, equal ping-pong buffers, a sub-batch with both a
 * replay cache and a CACHE, a missing table without a CACHE, a CACHE view
 * fc_cache_search would reject), creates the streams and
 * events and returns the executor in *out.  FC_ERR_CUDA if a stream or
 * event cannot be created (nothing is left allocated). */
fc_status fc_pipeline_create(const fc_pipeline_desc* desc, fc_pipeline** out);

/*
 * Enqueues one step of every sub-batch.  Per-step inputs are batch-wide
 * device arrays; sub-batch h reads its rows from `first`:
 *   d_q [B][n_pad][H][D] bf16, d_k_tree and d_v_tree [B][Hkv][n_pad][D]
 *   bf16 (unrotated when rope_base > 0), d_want_hit [B] (NULL: every query
 *   may hit the replay cache), d_plen [B], d_rtok [B][n_pad] (the synthetic
 *   model's draws).
 * phase (0 or 1) selects the ping-pong lengths read; alternate it.  flags:
 * 0, or FC_PIPELINE_NO_ATTENTION to leave out the attention launch (the
 * synthetic predictions do not read its output; d_q may then be NULL).  Every
 * sub-batch first waits for the work enqueued on `caller`; `caller` does not
 * wait for the sub-batches (fc_pipeline_join does).  stage_events: NULL, or
 * [n_parts][4][2] cudaEvent_t (NULL entries skipped) recorded at the start
 * and end of the retrieval, tree, attention and verification stages.  A
 * non-OK status from an entry point is returned at once, and the
 * sub-batches' later launches of this step are not enqueued.
 */
#define FC_PIPELINE_NO_ATTENTION 1
fc_status fc_pipeline_step(fc_pipeline* pl, int phase, int flags, const void* d_q, const void* d_k_tree,
                           const void* d_v_tree, const int32_t* d_want_hit, const int32_t* d_plen,
                           const uint32_t* d_rtok, fc_stream caller, void* const* stage_events);

/* fc_pipeline_step for sub-batch `part` alone: its work waits for the work
 * enqueued on `caller` and then runs on its own streams; the other
 * sub-batches are untouched.  With it each sub-batch can be captured into a
 * CUDA graph of its own, so that replays never join the sub-batches.
 * stage_events as fc_pipeline_step's (entries of other sub-batches unused). */
fc_status fc_pipeline_step_part(fc_pipeline* pl, int part, int phase, int flags, const void* d_q,
                                const void* d_k_tree, const void* d_v_tree, const int32_t* d_want_hit,
                                const int32_t* d_plen, const uint32_t* d_rtok, fc_stream caller,
                                void* const* stage_events);

/* `caller` waits for everything enqueued on sub-batch `part`'s streams. */
fc_status fc_pipeline_join_part(fc_pipeline* pl, int part, fc_stream caller);

/* Waits for sub-batch `part`'s work enqueued so far, then returns and clears
 * its error word: the most severe device-detected error its kernels recorded
 * (FC_OK if none).  With a word per sub-batch an error is reported for the
 * sub-batch that raised it, whatever the other sub-batches' streams do.
 * FC_ERR_INVALID_ARG if the sub-batch was created without a word.
 * Synchronous. */
fc_status fc_pipeline_error(fc_pipeline* pl, int part);

/* The stream that runs sub-batch `part`'s chain (lookup .. append; the
 * attention runs on a second stream and rejoins it before the predictions),
 * or NULL for a bad argument.  Work the caller enqueues there runs after
 * the sub-batch's steps enqueued so far, e.g. reading its results back. */
fc_stream fc_pipeline_stream(const fc_pipeline* pl, int part);

/* `caller` waits for everything enqueued on the sub-batches' streams. */
fc_status fc_pipeline_join(fc_pipeline* pl, fc_stream caller);

/*
 * A CUDA graph of n_steps consecutive steps of sub-batch `part`, captured
 * from its streams: step t reads phase (phase0 + t) & 1 and the inputs
 * d_q[t], d_k_tree[t], d_v_tree[t], d_want_hit[t] (d_want_hit itself may be
 * NULL), d_plen[t], d_rtok[t] (host arrays of n_steps device pointers, each
 * as fc_pipeline_step's; d_q may be NULL with FC_PIPELINE_NO_ATTENTION).
 * Every kernel node keeps the priority of the stream it runs on in the eager
 * step (the chain above the attention), and the graph is instantiated to run
 * by those node priorities, whatever stream it is launched into.  The graph
 * is uploaded to the device on the sub-batch's chain stream, so that its
 * first launch does not pay for it.  Capturing enqueues no kernel: the
 * sub-batch's state advances by n_steps at each launch,
 * so launch graphs whose phases continue the sub-batch's.  The graph holds
 * the pointers it was captured with; it must not outlive them or the
 * executor.  FC_ERR_INVALID_ARG for a bad argument, FC_ERR_CUDA if the
 * capture or instantiation fails (nothing is left allocated).
 */
typedef struct fc_pipeline_graph fc_pipeline_graph;
fc_status fc_pipeline_capture_part(fc_pipeline* pl, int part, int n_steps, int phase0, int flags,
                                   const void* const* d_q, const void* const* d_k_tree,
                                   const void* const* d_v_tree, const int32_t* const* d_want_hit,
                                   const int32_t* const* d_plen, const uint32_t* const* d_rtok,
                                   fc_pipeline_graph** out);

/* Launches the graph into `s`: it runs after the work already enqueued on s,
 * and s's later work runs after it. */
fc_status fc_pipeline_graph_launch(fc_pipeline_graph* g, fc_stream s);

/* Counts the graph's kernel nodes by priority: *n_chain at the chain
 * stream's, *n_attn at the attention stream's (FC_ERR_INTERNAL if a node
 * has another). */
fc_status fc_pipeline_graph_kernels(const fc_pipeline_graph* g, int* n_chain, int* n_attn);

/* Frees the graph (NULL is ignored); launches already made still run. */
void fc_pipeline_graph_destroy(fc_pipeline_graph* g);

/* Waits for the executor's streams, then frees its streams and events. */
void fc_pipeline_destroy(fc_pipeline* pl);

#ifdef __cplusplus
}
#endif

#endif /* FASTCODER_H_ */

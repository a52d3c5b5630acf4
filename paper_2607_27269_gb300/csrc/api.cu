// The C ABI of libgbmla.so (include/gbmla.h): host-side argument checks,
// split resolution, the per-device status word and the launches.
#include <math.h>
#include <stdlib.h>
#include <string.h>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace gbmla {
namespace {

// Sticky status word, one per device (a __device__ variable lives once per
// device context).  Kernels receive its device address.
__device__ unsigned g_status_word;

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
unsigned *g_status_ptr[kMaxDevices];
int g_sm_count[kMaxDevices];

// Device address of this device's status word and its SM count, looked up
// once per device with that device current.
mla_status device_info(unsigned **status, int *sms)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return MLA_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_status_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return MLA_ERR_CUDA;
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return MLA_ERR_CUDA;
        g_status_ptr[dev] = static_cast<unsigned *>(p);
        g_sm_count[dev] = n;
    }
    if (status) *status = g_status_ptr[dev];
    if (sms) *sms = g_sm_count[dev];
    return MLA_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

mla_status check_dims(const mla_dims *d)
{
    if (!d) return MLA_ERR_INVALID_ARG;
    if (d->num_heads <= 0 || d->num_kv_groups <= 0 || d->num_heads % d->num_kv_groups) return MLA_ERR_INVALID_ARG;
    if (d->d_nope <= 0 || d->d_v <= 0 || d->rank <= 0 || d->d_rope < 0 || d->hidden < 0) return MLA_ERR_INVALID_ARG;
    if (!(d->sm_scale > 0.f) || !isfinite(d->sm_scale)) return MLA_ERR_INVALID_ARG;
    if (!(d->rope_base > 1.f) || !isfinite(d->rope_base)) return MLA_ERR_INVALID_ARG;
    if (d->rope_style != 0 && d->rope_style != 1) return MLA_ERR_INVALID_ARG;
    if (d->d_rope != 32 && d->d_rope != 64) return MLA_ERR_UNSUPPORTED;
    if (d->rank % 64 || d->rank > 512) return MLA_ERR_UNSUPPORTED;
    if (d->d_nope % 8 || d->d_nope > 256 || d->d_v % 8 || d->d_v > 256) return MLA_ERR_UNSUPPORTED;
    if (d->num_heads > 128) return MLA_ERR_UNSUPPORTED;
    return MLA_OK;
}

mla_status check_cache(const mla_dims *d, const mla_cache *c, CacheView *v)
{
    if (!c || !c->c_kv || !c->k_rope) return MLA_ERR_INVALID_ARG;
    if (!aligned16(c->c_kv) || !aligned16(c->k_rope)) return MLA_ERR_INVALID_ARG;
    if (c->c_tok_stride % 8 || c->r_tok_stride % 8 || c->c_blk_stride % 8 || c->r_blk_stride % 8)
        return MLA_ERR_INVALID_ARG;
    if (c->c_tok_stride < d->rank || c->r_tok_stride < d->d_rope || c->c_blk_stride < 0 || c->r_blk_stride < 0)
        return MLA_ERR_INVALID_ARG;
    if (c->capacity <= 0) return MLA_ERR_INVALID_ARG;
    if (c->block_table) {
        if (c->page_size != 64) return MLA_ERR_UNSUPPORTED;
        if (c->num_pages <= 0 || c->bt_stride <= 0) return MLA_ERR_INVALID_ARG;
        if (static_cast<int64_t>(c->bt_stride) * c->page_size < c->capacity) return MLA_ERR_INVALID_ARG;
    }
    v->c_kv = c->c_kv;
    v->k_rope = c->k_rope;
    v->c_tok = c->c_tok_stride;
    v->r_tok = c->r_tok_stride;
    v->c_blk = c->c_blk_stride;
    v->r_blk = c->r_blk_stride;
    v->block_table = c->block_table;
    v->bt_stride = c->bt_stride;
    v->page_size = c->page_size;
    v->num_pages = c->num_pages;
    v->capacity = c->capacity;
    return MLA_OK;
}

// The tensor-core kernel serves every shape with rank % 128 == 0; the
// CUDA-core kernel serves the rest.  The attn_simt testing aid forces the
// CUDA-core kernel (used by tests that compare the two).
bool use_tc_kernel(const mla_dims *d)
{
    if (tuning().attn_simt) return false;
    return d->rank % 128 == 0;
}

// Partitions used for (dims, batch, q_len, max_kv_len): `requested` if > 0,
// otherwise enough partitions that the query groups fill the SMs (one CTA per
// SM for the tensor-core kernel, two for the CUDA-core kernel), never more
// partitions than tiles.
int resolve_splits(const mla_dims *d, int batch, int q_len, int max_kv_len, int requested, int sms)
{
    const int64_t max_tiles = static_cast<int64_t>(batch) * ((max_kv_len + MLA_SPLIT_TILE - 1) / MLA_SPLIT_TILE);
    if (requested > 0) return requested;
    const int rows = q_len * d->num_heads;
    int64_t s;
    if (use_tc_kernel(d)) {
        s = sms / attn_tc_shape(rows).groups;  // one CTA per SM
    } else {
        const int groups = (rows + kSimtRows - 1) / kSimtRows;
        s = (2 * static_cast<int64_t>(sms) + groups - 1) / groups;
    }
    if (s > max_tiles) s = max_tiles;
    if (s < 1) s = 1;
    // Short partitions (at most four tiles each, with the tile count bounded
    // by batch x max_kv_len): the fewest partitions that keep the same most
    // tiles per partition, since every partition adds partials for the combine
    // to merge (qwen-like batches: 152 -> 128 partitions of 2 tiles cut the
    // attention + combine from 22.3 to 16.9 us).  Longer ones keep one per SM:
    // with ragged lengths the bound is loose and the idle SMs would cost more.
    const int64_t per = (max_tiles + s - 1) / s;
    if (per <= 4) s = (max_tiles + per - 1) / per;
    return static_cast<int>(s);
}

thread_local cudaError_t g_last_cuda_error = cudaSuccess;

Tuning g_tuning;
std::once_flag g_tuning_once;

int env_int(const char *name)
{
    const char *v = getenv(name);
    return v ? atoi(v) : 0;
}

void read_tuning()
{
    Tuning t;
    const char *k = getenv("GBMLA_ATTN_KERNEL");
    t.attn_simt = (k && strcmp(k, "simt") == 0) ? 1 : 0;
    t.tc_max_rows = env_int("GBMLA_TC_MAX_N");
    t.tc_max_slots = env_int("GBMLA_TC_MAX_SLOTS");
    t.tc_pv_slots = env_int("GBMLA_TC_PV_SLOTS");
    const char *ab = getenv("GBMLA_ABSORB");
    t.absorb_path = !ab ? 0 : strcmp(ab, "persistent") == 0 ? 1 : strcmp(ab, "gemm") == 0 ? 2 : 0;
    const char *tq = getenv("GBMLA_TC_QUERY");
    t.tc_query = !tq ? 0 : strcmp(tq, "resident") == 0 ? 1 : strcmp(tq, "streamed") == 0 ? 2 : 0;
    std::lock_guard<std::mutex> lock(g_mutex);
    g_tuning = t;
}

// Scratch of mla_decode_attn_noalloc: the split partials live here instead of
// in caller buffers.  32 MiB, reserved on every device that loads the library
// for as long as the process lives.  Host code cannot use the symbol's name as
// a device address; noalloc_scratch() looks the address up per device.
constexpr size_t kNoallocScratchFloats = (size_t{32} << 20) / sizeof(float);
static __device__ __align__(256) float g_noalloc_scratch[kNoallocScratchFloats];
float *g_noalloc_ptr[kMaxDevices];

// Device address of this device's scratch array, looked up once per device
// with that device current (a host-side query; nothing is allocated).
mla_status noalloc_scratch(float **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return MLA_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_noalloc_ptr[dev]) {
        void *p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) {
            g_last_cuda_error = e;
            return MLA_ERR_CUDA;
        }
        g_noalloc_ptr[dev] = static_cast<float *>(p);
    }
    *out = g_noalloc_ptr[dev];
    return MLA_OK;
}

mla_status from_cuda(cudaError_t e)
{
    if (e == cudaSuccess) return MLA_OK;
    g_last_cuda_error = e;
    return MLA_ERR_CUDA;
}

__global__ void selftest_wait_kernel(uint64_t limit_ns, unsigned *status)
{
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) mbar_init(&bar, 1);
    __syncthreads();
    // Nothing arrives on `bar`: the bounded wait must give up.
    if (!mbar_wait(smem_u32(&bar), 0, limit_ns)) {
        if (threadIdx.x == 0) record_status(status, kStatusTimeout);
    }
}

}  // namespace

const Tuning &tuning()
{
    std::call_once(g_tuning_once, read_tuning);
    return g_tuning;
}

void reload_tuning()
{
    std::call_once(g_tuning_once, read_tuning);
    read_tuning();
}

cudaError_t launch_selftest_wait(int64_t limit_ns, unsigned *status, cudaStream_t st)
{
    selftest_wait_kernel<<<1, 32, 0, st>>>(static_cast<uint64_t>(limit_ns), status);
    return cudaGetLastError();
}

}  // namespace gbmla

using namespace gbmla;

// The five entry points of the step, each as validation followed by the
// launch; with launch == false they only validate (mla_decode_step checks
// every stage before it launches any).
namespace {

mla_status mla_cache_append_impl(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t n_new,
                                 const void *c_new, const void *kr_new, const int32_t *start_pos, void *stream, bool launch)
{
    mla_status s = check_dims(dims);
    if (s != MLA_OK) return s;
    CacheView v;
    if ((s = check_cache(dims, cache, &v)) != MLA_OK) return s;
    if (batch < 0 || n_new < 0 || batch > 65535 || n_new > 65535) return MLA_ERR_INVALID_ARG;
    if (batch == 0 || n_new == 0) return MLA_OK;
    if (!c_new || !kr_new || !start_pos || !aligned16(c_new)) return MLA_ERR_INVALID_ARG;
    if (!launch) return MLA_OK;  // (validation only)
    unsigned *status = nullptr;
    if ((s = device_info(&status, nullptr)) != MLA_OK) return s;
    return from_cuda(launch_append(*dims, v, batch, n_new, c_new, kr_new, start_pos, status,
                                   static_cast<cudaStream_t>(stream)));
}

mla_status mla_absorb_q_impl(const mla_dims *dims, int32_t batch, int32_t q_len, const void *q_nope,
                             const void *q_pe, const int32_t *kv_len, const void *w_uk, void *q_abs, void *stream, bool launch)
{
    mla_status s = check_dims(dims);
    if (s != MLA_OK) return s;
    if (batch < 0 || q_len < 1 || q_len > 16) return MLA_ERR_INVALID_ARG;
    if (batch == 0) return MLA_OK;
    if (!q_nope || !q_pe || !kv_len || !w_uk || !q_abs) return MLA_ERR_INVALID_ARG;
    if (!aligned16(q_nope) || !aligned16(w_uk) || !aligned16(q_abs)) return MLA_ERR_INVALID_ARG;
    if (static_cast<int64_t>(batch) * q_len > (1 << 30)) return MLA_ERR_UNSUPPORTED;
    if (!launch) return MLA_OK;  // (validation only)
    unsigned *status = nullptr;
    if ((s = device_info(&status, nullptr)) != MLA_OK) return s;
    return from_cuda(launch_absorb(*dims, batch, q_len, q_nope, q_pe, kv_len, w_uk, q_abs, status,
                                   static_cast<cudaStream_t>(stream)));
}

mla_status mla_decode_attn_impl(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t q_len,
                                const int32_t *kv_len, int32_t max_kv_len, const void *q_abs, int32_t num_splits,
                                float *o_part, float *lse_part, void *stream, bool launch, float *o_final = nullptr,
                                float *lse_final = nullptr)
{
    mla_status s = check_dims(dims);
    if (s != MLA_OK) return s;
    CacheView v;
    if ((s = check_cache(dims, cache, &v)) != MLA_OK) return s;
    if (batch < 0 || q_len < 1 || q_len > 16 || num_splits < 0 || num_splits > 65535) return MLA_ERR_INVALID_ARG;
    if (max_kv_len < q_len || max_kv_len > cache->capacity) return MLA_ERR_INVALID_ARG;
    if (batch == 0) return MLA_OK;
    if (!kv_len || !q_abs || !o_part || !lse_part || !aligned16(o_part) || !aligned16(q_abs))
        return MLA_ERR_INVALID_ARG;
    if (!launch) return MLA_OK;  // (validation only)
    unsigned *status = nullptr;
    int sms = 0;
    if ((s = device_info(&status, &sms)) != MLA_OK) return s;
    AttnArgs a;
    a.batch = batch;
    a.q_len = q_len;
    a.num_heads = dims->num_heads;
    a.rank = dims->rank;
    a.d_rope = dims->d_rope;
    a.sm_scale = dims->sm_scale;
    a.kv_len = kv_len;
    a.max_kv = max_kv_len;
    a.q_abs = q_abs;
    a.num_splits = resolve_splits(dims, batch, q_len, max_kv_len, num_splits, sms);
    a.o_part = o_part;
    a.lse_part = lse_part;
    a.o_final = o_final;
    a.lse_final = lse_final;
    a.cache = v;
    a.status = status;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    return from_cuda(use_tc_kernel(dims) ? launch_attn_tc(a, st) : launch_attn_simt(a, st));
}

mla_status mla_combine_impl(const mla_dims *dims, int32_t batch, int32_t q_len, int32_t num_splits,
                            const int32_t *kv_len, int32_t max_kv_len, const float *o_part, const float *lse_part,
                            float *o_lat, float *lse, void *stream, bool launch, bool skip_whole = false)
{
    mla_status s = check_dims(dims);
    if (s != MLA_OK) return s;
    if (batch < 0 || q_len < 1 || q_len > 16 || num_splits < 0 || max_kv_len < q_len) return MLA_ERR_INVALID_ARG;
    if (batch == 0) return MLA_OK;
    if (!kv_len || !o_part || !lse_part || !o_lat || !aligned16(o_part) || !aligned16(o_lat))
        return MLA_ERR_INVALID_ARG;
    if (!launch) return MLA_OK;  // (validation only)
    int sms = 0;
    if ((s = device_info(nullptr, &sms)) != MLA_OK) return s;
    const int S = resolve_splits(dims, batch, q_len, max_kv_len, num_splits, sms);
    // a length above max_kv_len counts as unusable in both kernels
    return from_cuda(launch_combine(batch, q_len, dims->num_heads, dims->rank, max_kv_len, S, kv_len, o_part,
                                    lse_part, o_lat, lse, static_cast<cudaStream_t>(stream), 1, skip_whole));
}

mla_status mla_out_proj_impl(const mla_dims *dims, int32_t batch, int32_t q_len, const float *o_lat,
                             const void *w_uv, const void *w_o, void *o, void *out, void *stream, bool launch)
{
    mla_status s = check_dims(dims);
    if (s != MLA_OK) return s;
    if (batch < 0 || q_len < 1 || q_len > 16) return MLA_ERR_INVALID_ARG;
    if (batch == 0) return MLA_OK;
    if (!o_lat || !w_uv || !o) return MLA_ERR_INVALID_ARG;
    if (w_o && dims->hidden > 0 && !out) return MLA_ERR_INVALID_ARG;
    if (!aligned16(o_lat) || !aligned16(w_uv) || !aligned16(o)) return MLA_ERR_INVALID_ARG;
    if (w_o && dims->hidden > 0 && (!aligned16(w_o) || !aligned16(out))) return MLA_ERR_INVALID_ARG;
    if (!launch) return MLA_OK;  // (validation only)
    unsigned *status = nullptr;
    if ((s = device_info(&status, nullptr)) != MLA_OK) return s;
    return from_cuda(launch_out_proj(*dims, batch, q_len, o_lat, w_uv, w_o, o, out, status,
                                     static_cast<cudaStream_t>(stream)));
}

}  // namespace

extern "C" {

const char *mla_status_str(mla_status s)
{
    switch (s) {
    case MLA_OK: return "MLA_OK";
    case MLA_ERR_INVALID_ARG: return "MLA_ERR_INVALID_ARG";
    case MLA_ERR_UNSUPPORTED: return "MLA_ERR_UNSUPPORTED";
    case MLA_ERR_CUDA: return "MLA_ERR_CUDA";
    case MLA_ERR_DEVICE_BOUNDS: return "MLA_ERR_DEVICE_BOUNDS";
    case MLA_ERR_DEVICE_TIMEOUT: return "MLA_ERR_DEVICE_TIMEOUT";
    }
    return "MLA_ERR_UNKNOWN";
}

mla_status mla_workspace_size(const mla_dims *dims, int32_t batch, int32_t q_len, int32_t max_kv_len,
                              int32_t num_splits, size_t *o_part_bytes, size_t *lse_part_bytes,
                              int32_t *num_splits_used)
{
    mla_status s = check_dims(dims);
    if (s != MLA_OK) return s;
    if (batch < 0 || q_len < 1 || q_len > 16 || max_kv_len < q_len || num_splits < 0) return MLA_ERR_INVALID_ARG;
    int sms = 0;
    if ((s = device_info(nullptr, &sms)) != MLA_OK) return s;
    const int S = resolve_splits(dims, batch, q_len, max_kv_len, num_splits, sms);
    const size_t slots = batch > 0 ? static_cast<size_t>(batch) + S - 1 : 0;
    const size_t rows = static_cast<size_t>(q_len) * dims->num_heads;
    if (o_part_bytes) *o_part_bytes = slots * rows * dims->rank * sizeof(float);
    if (lse_part_bytes) *lse_part_bytes = slots * rows * sizeof(float);
    if (num_splits_used) *num_splits_used = S;
    return MLA_OK;
}

mla_status mla_cache_append(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t n_new,
                            const void *c_new, const void *kr_new, const int32_t *start_pos, void *stream)
{
    return mla_cache_append_impl(dims, cache, batch, n_new, c_new, kr_new, start_pos, stream, true);
}

mla_status mla_project_append(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t n_new,
                              const void *h, const void *w_dkv, const void *w_kr, const void *w_q,
                              const int32_t *start_pos, void *q_nope, void *q_pe, void *stream)
{
    mla_status s = check_dims(dims);
    if (s != MLA_OK) return s;
    CacheView v;
    if ((s = check_cache(dims, cache, &v)) != MLA_OK) return s;
    if (batch < 0 || n_new < 0 || batch > 65535 || n_new > 65535) return MLA_ERR_INVALID_ARG;
    if (dims->hidden <= 0 || dims->hidden % 8) return MLA_ERR_INVALID_ARG;
    if (batch == 0 || n_new == 0) return MLA_OK;
    if (!h || !w_dkv || !w_kr || !start_pos) return MLA_ERR_INVALID_ARG;
    if (!aligned16(h) || !aligned16(w_dkv) || !aligned16(w_kr)) return MLA_ERR_INVALID_ARG;
    if (w_q && (!q_nope || !q_pe || !aligned16(w_q) || !aligned16(q_nope) || !aligned16(q_pe)))
        return MLA_ERR_INVALID_ARG;
    if (static_cast<int64_t>(batch) * n_new > (1 << 24)) return MLA_ERR_UNSUPPORTED;
    unsigned *status = nullptr;
    if ((s = device_info(&status, nullptr)) != MLA_OK) return s;
    return from_cuda(launch_project(*dims, v, batch, n_new, h, w_dkv, w_kr, w_q, start_pos, q_nope, q_pe, status,
                                    static_cast<cudaStream_t>(stream)));
}

mla_status mla_acceptance_stats(int32_t rows, int32_t vocab, int32_t logits_dtype, const void *draft_logits,
                                const void *target_logits, int64_t row_stride, float *alpha_sample,
                                int32_t *argmax_draft, int32_t *argmax_target, int32_t *greedy_accept, void *stream)
{
    if (rows < 0 || rows > 65535 || vocab <= 0 || row_stride < vocab) return MLA_ERR_INVALID_ARG;
    if (logits_dtype != 0 && logits_dtype != 1) return MLA_ERR_INVALID_ARG;
    if (rows == 0) return MLA_OK;
    const int64_t es = logits_dtype == 0 ? 4 : 2;
    if (!draft_logits || !target_logits || !aligned16(draft_logits) || !aligned16(target_logits) ||
        (row_stride * es) % 16)
        return MLA_ERR_INVALID_ARG;
    unsigned *status = nullptr;
    mla_status s = device_info(&status, nullptr);
    if (s != MLA_OK) return s;
    return from_cuda(launch_acceptance(rows, vocab, logits_dtype, draft_logits, target_logits, row_stride,
                                       alpha_sample, argmax_draft, argmax_target, greedy_accept, status,
                                       static_cast<cudaStream_t>(stream)));
}

// ---- original GQA
namespace {
// The GQA layer seen through the MLA checks: values where the latent goes,
// keys where the positional keys go.
mla_status gqa_as_mla(const mla_gqa_dims *g, mla_dims *d)
{
    if (!g || g->num_heads <= 0 || g->num_kv_groups <= 0 || g->num_heads % g->num_kv_groups)
        return MLA_ERR_INVALID_ARG;
    if (!(g->sm_scale > 0.f) || !isfinite(g->sm_scale) || !(g->rope_base > 1.f) || !isfinite(g->rope_base))
        return MLA_ERR_INVALID_ARG;
    if (g->rope_style != 0 && g->rope_style != 1) return MLA_ERR_INVALID_ARG;
    if (g->head_dim != 64 && g->head_dim != 128) return MLA_ERR_UNSUPPORTED;
    *d = mla_dims{g->num_heads, g->num_kv_groups, g->head_dim, g->head_dim, g->head_dim, g->head_dim, 0,
                  g->sm_scale, g->rope_style, g->rope_base};
    return MLA_OK;
}

int gqa_splits(const mla_gqa_dims *g, int batch, int max_kv_len, int requested, int sms)
{
    if (requested > 0) return requested;
    int64_t s = sms;  // one CTA per SM
    const int64_t tiles = static_cast<int64_t>(batch) * g->num_kv_groups * ((max_kv_len + MLA_SPLIT_TILE - 1) / MLA_SPLIT_TILE);
    if (s > tiles) s = tiles;
    if (s < 1) s = 1;
    const int64_t per = (tiles + s - 1) / s;  // short partitions: the fewest with the same most tiles each
    if (per <= 4) s = (tiles + per - 1) / per;
    return static_cast<int>(s);
}
}  // namespace

mla_status mla_gqa_append(const mla_gqa_dims *dims, const mla_cache *cache, int32_t batch, int32_t n_new,
                          const void *k_new, const void *v_new, const int32_t *start_pos, void *stream)
{
    mla_dims d;
    mla_status s = gqa_as_mla(dims, &d);
    if (s != MLA_OK) return s;
    CacheView v;
    if ((s = check_cache(&d, cache, &v)) != MLA_OK) return s;
    if (batch < 0 || n_new < 0 || static_cast<int64_t>(batch) * dims->num_kv_groups > 65535 || n_new > 65535)
        return MLA_ERR_INVALID_ARG;
    if (batch == 0 || n_new == 0) return MLA_OK;
    if (!k_new || !v_new || !start_pos || !aligned16(v_new)) return MLA_ERR_INVALID_ARG;
    unsigned *status = nullptr;
    if ((s = device_info(&status, nullptr)) != MLA_OK) return s;
    return from_cuda(launch_append(d, v, batch * dims->num_kv_groups, n_new, v_new, k_new, start_pos, status,
                                   static_cast<cudaStream_t>(stream), dims->num_kv_groups));
}

mla_status mla_gqa_workspace_size(const mla_gqa_dims *dims, int32_t batch, int32_t q_len, int32_t max_kv_len,
                                  int32_t num_splits, size_t *o_part_bytes, size_t *lse_part_bytes,
                                  int32_t *num_splits_used)
{
    mla_dims d;
    mla_status s = gqa_as_mla(dims, &d);
    if (s != MLA_OK) return s;
    if (batch < 0 || q_len < 1 || q_len > 16 || max_kv_len < q_len || num_splits < 0) return MLA_ERR_INVALID_ARG;
    if (q_len * (dims->num_heads / dims->num_kv_groups) > 128) return MLA_ERR_UNSUPPORTED;
    int sms = 0;
    if ((s = device_info(nullptr, &sms)) != MLA_OK) return s;
    const int S = gqa_splits(dims, batch, max_kv_len, num_splits, sms);
    const size_t units = static_cast<size_t>(batch) * dims->num_kv_groups;
    const size_t slots = units > 0 ? units + S - 1 : 0;
    const size_t rows = static_cast<size_t>(q_len) * (dims->num_heads / dims->num_kv_groups);
    if (o_part_bytes) *o_part_bytes = slots * rows * dims->head_dim * sizeof(float);
    if (lse_part_bytes) *lse_part_bytes = slots * rows * sizeof(float);
    if (num_splits_used) *num_splits_used = S;
    return MLA_OK;
}

mla_status mla_gqa_decode_attn(const mla_gqa_dims *dims, const mla_cache *cache, int32_t batch, int32_t q_len,
                               const int32_t *kv_len, int32_t max_kv_len, const void *q, int32_t num_splits,
                               float *o_part, float *lse_part, float *o, float *lse, void *stream)
{
    mla_dims d;
    mla_status s = gqa_as_mla(dims, &d);
    if (s != MLA_OK) return s;
    CacheView v;
    if ((s = check_cache(&d, cache, &v)) != MLA_OK) return s;
    if (batch < 0 || q_len < 1 || q_len > 16 || num_splits < 0 || num_splits > 65535) return MLA_ERR_INVALID_ARG;
    if (static_cast<int64_t>(batch) * dims->num_kv_groups > 65535) return MLA_ERR_UNSUPPORTED;
    if (max_kv_len < q_len || max_kv_len > cache->capacity) return MLA_ERR_INVALID_ARG;
    const int hpg = dims->num_heads / dims->num_kv_groups;
    if (q_len * hpg > 128) return MLA_ERR_UNSUPPORTED;
    if (batch == 0) return MLA_OK;
    if (!kv_len || !q || !o_part || !lse_part || !o || !aligned16(q) || !aligned16(o_part) || !aligned16(o))
        return MLA_ERR_INVALID_ARG;
    unsigned *status = nullptr;
    int sms = 0;
    if ((s = device_info(&status, &sms)) != MLA_OK) return s;
    GqaLaunch g;
    g.batch = batch;
    g.q_len = q_len;
    g.groups = dims->num_kv_groups;
    g.hpg = hpg;
    g.head_dim = dims->head_dim;
    g.max_kv = max_kv_len;
    g.num_splits = gqa_splits(dims, batch, max_kv_len, num_splits, sms);
    g.sm_scale = dims->sm_scale;
    g.rope_style = dims->rope_style;
    g.rope_base = dims->rope_base;
    g.kv_len = kv_len;
    g.q = q;
    g.o_part = o_part;
    g.lse_part = lse_part;
    g.status = status;
    g.cache = v;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e = launch_gqa_attn(g, st);
    if (e != cudaSuccess) return from_cuda(e);
    return from_cuda(launch_combine(batch * g.groups, q_len, hpg, dims->head_dim, max_kv_len, g.num_splits, kv_len,
                                    o_part, lse_part, o, lse, st, g.groups));
}

mla_status mla_gqa_project(const mla_gqa_dims *dims, int32_t batch, int32_t n_new, int32_t hidden, const void *h,
                           const void *w_q, const void *w_k, const void *w_v, void *q, void *k_new, void *v_new,
                           void *stream)
{
    mla_dims d;
    mla_status s = gqa_as_mla(dims, &d);
    if (s != MLA_OK) return s;
    if (batch < 0 || n_new < 0 || hidden <= 0 || hidden % 8) return MLA_ERR_INVALID_ARG;
    if (batch == 0 || n_new == 0) return MLA_OK;
    const void *ptrs[7] = {h, w_q, w_k, w_v, q, k_new, v_new};
    for (const void *p : ptrs)
        if (!p || !aligned16(p)) return MLA_ERR_INVALID_ARG;
    if (static_cast<int64_t>(batch) * n_new > (1 << 24)) return MLA_ERR_UNSUPPORTED;
    unsigned *status = nullptr;
    if ((s = device_info(&status, nullptr)) != MLA_OK) return s;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int M = batch * n_new, hd = dims->head_dim;
    const int cols[3] = {dims->num_heads * hd, dims->num_kv_groups * hd, dims->num_kv_groups * hd};
    const void *w[3] = {w_q, w_k, w_v};
    void *outs[3] = {q, k_new, v_new};
    for (int k = 0; k < 3; ++k) {
        GroupGemm p;
        p.M = M;
        p.N = cols[k];
        p.K = hidden;
        p.G = 1;
        p.hpg = 1;
        p.blk = 1;
        p.A = h;
        p.a_f32 = 0;
        p.lda = hidden;
        p.B = w[k];
        p.b_nmajor = 0;
        p.C = outs[k];
        p.ldc = cols[k];
        p.status = status;
        const cudaError_t e = launch_group_gemm(p, st);
        if (e != cudaSuccess) return from_cuda(e);
    }
    return MLA_OK;
}

mla_status mla_gqa_out_proj(const mla_gqa_dims *dims, int32_t batch, int32_t q_len, int32_t hidden, const float *o,
                            const void *w_o, void *out, void *stream)
{
    mla_dims d;
    mla_status s = gqa_as_mla(dims, &d);
    if (s != MLA_OK) return s;
    if (batch < 0 || q_len < 0 || hidden <= 0 || hidden % 8) return MLA_ERR_INVALID_ARG;
    if (batch == 0 || q_len == 0) return MLA_OK;
    if (!o || !w_o || !out || !aligned16(o) || !aligned16(w_o) || !aligned16(out)) return MLA_ERR_INVALID_ARG;
    unsigned *status = nullptr;
    if ((s = device_info(&status, nullptr)) != MLA_OK) return s;
    GroupGemm p;
    p.M = batch * q_len;
    p.N = hidden;
    p.K = dims->num_heads * dims->head_dim;
    p.G = 1;
    p.hpg = 1;
    p.blk = 1;
    p.A = o;
    p.a_f32 = 1;
    p.lda = p.K;
    p.B = w_o;
    p.b_nmajor = 0;
    p.C = out;
    p.ldc = hidden;
    p.status = status;
    return from_cuda(launch_group_gemm(p, static_cast<cudaStream_t>(stream)));
}

mla_status mla_e2e_loss(int32_t rows, int32_t hidden, const void *a_mla, const void *a_orig, const uint8_t *mask,
                        float *loss, void *stream)
{
    if (rows < 0 || hidden <= 0 || hidden % 8 || !loss) return MLA_ERR_INVALID_ARG;
    if (rows > 0 && (!a_mla || !a_orig || !aligned16(a_mla) || !aligned16(a_orig))) return MLA_ERR_INVALID_ARG;
    return from_cuda(launch_e2e_loss(rows, hidden, a_mla, a_orig, mask, loss, static_cast<cudaStream_t>(stream)));
}

mla_status mla_absorb_q(const mla_dims *dims, int32_t batch, int32_t q_len, const void *q_nope, const void *q_pe,
                        const int32_t *kv_len, const void *w_uk, void *q_abs, void *stream)
{
    return mla_absorb_q_impl(dims, batch, q_len, q_nope, q_pe, kv_len, w_uk, q_abs, stream, true);
}

mla_status mla_decode_attn(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t q_len,
                           const int32_t *kv_len, int32_t max_kv_len, const void *q_abs, int32_t num_splits,
                           float *o_part, float *lse_part, void *stream)
{
    return mla_decode_attn_impl(dims, cache, batch, q_len, kv_len, max_kv_len, q_abs, num_splits, o_part, lse_part,
                                stream, true);
}

mla_status mla_combine(const mla_dims *dims, int32_t batch, int32_t q_len, int32_t num_splits,
                       const int32_t *kv_len, int32_t max_kv_len, const float *o_part, const float *lse_part,
                       float *o_lat, float *lse, void *stream)
{
    return mla_combine_impl(dims, batch, q_len, num_splits, kv_len, max_kv_len, o_part, lse_part, o_lat, lse, stream,
                            true);
}

mla_status mla_out_proj(const mla_dims *dims, int32_t batch, int32_t q_len, const float *o_lat, const void *w_uv,
                        const void *w_o, void *o, void *out, void *stream)
{
    return mla_out_proj_impl(dims, batch, q_len, o_lat, w_uv, w_o, o, out, stream, true);
}

mla_status mla_decode_step(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t q_len,
                           const void *c_new, const void *kr_new, const int32_t *start_pos, const void *q_nope,
                           const void *q_pe, const int32_t *kv_len, int32_t max_kv_len, const void *w_uk,
                           const void *w_uv, const void *w_o, int32_t num_splits, void *q_abs, float *o_part,
                           float *lse_part, float *o_lat, float *lse, void *o, void *out, void *stream)
{
    // A sequence whose tiles all fall in one partition has a one-slot merge,
    // which only copies: the tensor-core attention writes its final rows into
    // o_lat / lse itself and the combine skips it (the same bits either way).
    const bool direct = dims && use_tc_kernel(dims) && lse != nullptr;
    for (int pass = 0; pass < 2; ++pass) {  // every stage validated, then every stage launched
        const bool go = pass == 1;
        mla_status s = MLA_OK;
        if (c_new) s = mla_cache_append_impl(dims, cache, batch, q_len, c_new, kr_new, start_pos, stream, go);
        if (s == MLA_OK) s = mla_absorb_q_impl(dims, batch, q_len, q_nope, q_pe, kv_len, w_uk, q_abs, stream, go);
        if (s == MLA_OK)
            s = mla_decode_attn_impl(dims, cache, batch, q_len, kv_len, max_kv_len, q_abs, num_splits, o_part,
                                     lse_part, stream, go, direct ? o_lat : nullptr, direct ? lse : nullptr);
        if (s == MLA_OK)
            s = mla_combine_impl(dims, batch, q_len, num_splits, kv_len, max_kv_len, o_part, lse_part, o_lat, lse,
                                 stream, go, direct);
        if (s == MLA_OK) s = mla_out_proj_impl(dims, batch, q_len, o_lat, w_uv, w_o, o, out, stream, go);
        if (s != MLA_OK) return s;
    }
    return MLA_OK;
}

mla_status mla_check_status(void *stream)
{
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return MLA_ERR_CUDA;
    unsigned *status = nullptr;
    mla_status s = device_info(&status, nullptr);
    if (s != MLA_OK) return s;
    unsigned word = 0;
    if (cudaMemcpy(&word, status, sizeof word, cudaMemcpyDeviceToHost) != cudaSuccess) return MLA_ERR_CUDA;
    if (word) {
        const unsigned zero = 0;
        if (cudaMemcpy(status, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess) return MLA_ERR_CUDA;
    }
    if (word & kStatusTimeout) return MLA_ERR_DEVICE_TIMEOUT;
    if (word & kStatusBounds) return MLA_ERR_DEVICE_BOUNDS;
    return MLA_OK;
}

mla_status mla_decode_attn_noalloc(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t q_len,
                                   const int32_t *kv_len, int32_t max_kv_len, const void *q_abs, int32_t num_splits,
                                   float *o_lat, float *lse, void *stream)
{
    mla_status s = check_dims(dims);
    if (s != MLA_OK) return s;
    CacheView v;
    if ((s = check_cache(dims, cache, &v)) != MLA_OK) return s;
    if (batch < 0 || q_len < 1 || q_len > 16 || num_splits < 0 || num_splits > 65535) return MLA_ERR_INVALID_ARG;
    if (max_kv_len < q_len || max_kv_len > cache->capacity) return MLA_ERR_INVALID_ARG;
    if (batch == 0) return MLA_OK;
    if (!kv_len || !q_abs || !o_lat || !aligned16(q_abs) || !aligned16(o_lat)) return MLA_ERR_INVALID_ARG;
    unsigned *status = nullptr;
    int sms = 0;
    if ((s = device_info(&status, &sms)) != MLA_OK) return s;
    // partials for B + S - 1 slots must fit the fixed scratch; an automatic
    // split count shrinks to fit, an explicit one that does not fit is refused
    const size_t rows = static_cast<size_t>(q_len) * dims->num_heads;
    const size_t per_slot = rows * dims->rank;
    auto need = [&](int S) {
        const size_t slots = static_cast<size_t>(batch) + S - 1;
        return slots * per_slot + ((slots * rows + 63) & ~size_t{63});
    };
    int S = resolve_splits(dims, batch, q_len, max_kv_len, num_splits, sms);
    if (need(S) > kNoallocScratchFloats) {
        if (num_splits > 0) return MLA_ERR_UNSUPPORTED;
        const int64_t slots_max = static_cast<int64_t>((kNoallocScratchFloats - 64) / (per_slot + rows));
        S = static_cast<int>(slots_max - batch + 1);
        while (S >= 1 && need(S) > kNoallocScratchFloats) --S;
        if (S < 1) return MLA_ERR_UNSUPPORTED;
    }
    float *scratch = nullptr;
    if ((s = noalloc_scratch(&scratch)) != MLA_OK) return s;
    const size_t slots = static_cast<size_t>(batch) + S - 1;
    float *o_part = scratch;
    float *lse_part = scratch + ((slots * per_slot + 63) & ~size_t{63});
    AttnArgs a;
    a.batch = batch;
    a.q_len = q_len;
    a.num_heads = dims->num_heads;
    a.rank = dims->rank;
    a.d_rope = dims->d_rope;
    a.sm_scale = dims->sm_scale;
    a.kv_len = kv_len;
    a.max_kv = max_kv_len;
    a.q_abs = q_abs;
    a.num_splits = S;
    a.o_part = o_part;
    a.lse_part = lse_part;
    a.cache = v;
    a.status = status;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if ((s = from_cuda(use_tc_kernel(dims) ? launch_attn_tc(a, st) : launch_attn_simt(a, st))) != MLA_OK) return s;
    return from_cuda(launch_combine(batch, q_len, dims->num_heads, dims->rank, max_kv_len, S, kv_len, o_part,
                                    lse_part, o_lat, lse, st));
}

const char *mla_last_error(void)
{
    return g_last_cuda_error == cudaSuccess ? "" : cudaGetErrorString(g_last_cuda_error);
}

void mla_reload_tuning(void) { reload_tuning(); }

mla_status mla_selftest_wait_timeout(int64_t limit_ns, void *stream)
{
    if (limit_ns < 1000) limit_ns = 1000;
    if (limit_ns > 1000000000) limit_ns = 1000000000;
    unsigned *status = nullptr;
    mla_status s = device_info(&status, nullptr);
    if (s != MLA_OK) return s;
    return from_cuda(launch_selftest_wait(limit_ns, status, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"

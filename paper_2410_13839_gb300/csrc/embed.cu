// embed.cu -- rows of the concatenated sequence (Sec. III-A): token embedding
// (phoneme table for the phoneme prefix, codec table for acoustic prompt and
// generated codes) plus the sinusoidal position of the row.
#include "common.cuh"
#include "kernels.cuh"

namespace mtp {
namespace {

__global__ void __launch_bounds__(256) embed_kernel(const EmbedArgs a) {
    __shared__ int s_tok, s_pos, s_act, s_phone;
    const int r = blockIdx.x, tid = threadIdx.x;
    TraceEnd trace_guard(a.trace);
    // The next kernels read the slot state before their own dependency wait, so
    // they may start only once this launch is past its wait (the kernel that
    // updates the slot state is then complete).
    pdl_wait();
    pdl_launch_dependents();
    trace_wait(a.trace);
    if (tid == 0) {
        int seq = -1, pos = 0, tok = 0, phone = 0, last = 0;
        if (a.mode == 0) {  // decode: row r is fed token j of slot seq_base + r / n
            const int b = a.seq_base + r / a.n_heads, j = r % a.n_heads;
            if (r < a.rows && b < a.slots) {  // the slot's state in one round of independent loads
                const int act = a.active[b], dn = a.done[b], np = a.n_pending[b], len = a.seq_len[b];
                const int t = a.pending[b * a.n_max + j];
                if (act && !dn && j < np) {
                    seq = b;
                    pos = len + j;
                    tok = t;
                    last = (j == np - 1);
                }
            }
        } else if (a.mode == 2) {  // prefill lane: the plan kernel chose slot and position
            if (r < a.rows) {
                seq = a.row_seq[a.row0 + r];
                if (seq >= 0) {
                    pos = a.row_pos[a.row0 + r];
                    tok = a.prompt[(size_t)seq * a.prompt_stride + pos];
                    phone = pos < a.prompt_nph[seq];
                }
            }
        } else {  // prefill chunk: positions p0 .. p0 + rows - 1 of one slot
            pos = a.p0 + r;
            if (r < a.rows && pos < a.total) {
                seq = a.slot;
                tok = a.prompt[(size_t)a.slot * a.prompt_stride + pos];
                phone = pos < a.n_ph;
                last = (pos == a.total - 1);
            }
        }
        if (seq >= 0 && (pos >= a.max_pos || tok < 0 || tok >= (phone ? a.phone_vocab : a.codec_vocab))) {
            atomicOr(a.err, ERR_BOUNDS);
            seq = -1;
        }
        if (a.mode != 2) {  // the lane's plan is already written
            a.row_seq[r] = seq;
            a.row_pos[r] = seq >= 0 ? pos : -1;
            a.row_last[r] = seq >= 0 ? last : 0;
        }
        s_act = seq >= 0;
        s_tok = tok;
        s_pos = pos;
        s_phone = phone;
    }
    __syncthreads();
    if (a.zero_buf)
        for (int i = tid; i < a.d; i += blockDim.x) a.zero_buf[(size_t)r * a.d + i] = 0.f;
    float* x = a.x + (size_t)r * a.d;
    if (!s_act) {
        for (int i = tid; i < a.d; i += blockDim.x) x[i] = 0.f;
        return;
    }
    const float* pe = a.pe + (size_t)s_pos * a.d;
    const void* table = s_phone ? a.tok_phone : a.tok_codec;
    for (int i = tid; i < a.d; i += blockDim.x) {
        float e;
        if (a.w_bf16) {
            const uint16_t bits = reinterpret_cast<const uint16_t*>(table)[(size_t)s_tok * a.d + i];
            e = __uint_as_float((uint32_t)bits << 16);
        } else {
            e = reinterpret_cast<const float*>(table)[(size_t)s_tok * a.d + i];
        }
        x[i] = e + pe[i];
    }
}

// PE[p, 2i] = sin(p * 10000^(-2i/d)), PE[p, 2i+1] = cos(same), in double, stored fp32.
__global__ void pe_kernel(float* pe, int max_ctx, int d) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)max_ctx * (d / 2)) return;
    const int p = (int)(idx / (d / 2)), i = (int)(idx % (d / 2));
    const double inv_freq = pow(10000.0, -2.0 * i / d);
    const double ang = (double)p * inv_freq;
    pe[(size_t)p * d + 2 * i] = (float)sin(ang);
    pe[(size_t)p * d + 2 * i + 1] = (float)cos(ang);
}

__global__ void convert_rows_kernel(const void* src, int src_bf16, float* dst, long long n) {
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    dst[i] = src_bf16 ? __uint_as_float((uint32_t)reinterpret_cast<const uint16_t*>(src)[i] << 16)
                      : reinterpret_cast<const float*>(src)[i];
}

__global__ void __launch_bounds__(1024) lane_plan_kernel(const LanePlanArgs a) {
    __shared__ int s_scan[1024];
    pdl_wait();  // the previous step's selection moved the slots' state
    pdl_launch_dependents();
    const int b = threadIdx.x;
    for (int i = threadIdx.x; i < a.capacity; i += blockDim.x) {
        a.row_seq[a.row0 + i] = -1;
        a.row_pos[a.row0 + i] = -1;
        a.row_last[a.row0 + i] = 0;
    }
    int left = 0, len = 0;
    if (b < a.slots && a.active[b] && !a.done[b]) {
        left = max(0, a.prompt_left[b]);
        len = a.seq_len[b];
    }
    const int demand = (left + a.rpg - 1) / a.rpg * a.rpg;
    s_scan[b] = demand;  // inclusive scan of the padded demands (Hillis-Steele)
    __syncthreads();
    for (int o = 1; o < (int)blockDim.x; o <<= 1) {
        const int add = b >= o ? s_scan[b - o] : 0;
        __syncthreads();
        s_scan[b] += add;
        __syncthreads();
    }
    const int start = s_scan[b] - demand;
    int take = 0;
    if (left > 0 && start < a.capacity) {
        take = min(left, a.capacity - start);
        for (int i = 0; i < take; ++i) {
            const int row = a.row0 + start + i;
            a.row_seq[row] = b;
            a.row_pos[row] = len + i;
            a.row_last[row] = (i == take - 1 && take == left) ? 1 : 0;
        }
        a.prompt_left[b] = left - take;
        a.seq_len[b] = len + take;
    }
    if (b < a.slots) a.lane_take[b] = take;
}

__global__ void slot_set_kernel(SlotSet s) {
    if (threadIdx.x != 0) return;
    pdl_wait();
    const int b = s.slot;
    if (s.set_len >= 0) s.seq_len[b] = s.set_len;
    if (s.set_pending >= 0) s.n_pending[b] = s.set_pending;
    if (s.set_remaining >= 0) s.remaining[b] = s.set_remaining;
    if (s.set_done >= 0) s.done[b] = s.set_done;
    if (s.set_active >= 0) s.active[b] = s.set_active;
    if (s.set_gen >= 0) s.gen_count[b] = s.set_gen;
    if (s.set_prompt_left >= 0 && s.prompt_left) s.prompt_left[b] = s.set_prompt_left;
    if (s.set_prompt_nph >= 0 && s.prompt_nph) s.prompt_nph[b] = s.set_prompt_nph;
}

}  // namespace

cudaError_t launch_embed(const EmbedArgs& a, cudaStream_t s, bool pdl) {
    cudaLaunchConfig_t cfg = {};
    // rows past a.rows (up to the next multiple of 8) are written inactive
    cfg.gridDim = dim3(a.rows > MAX_ROWS ? (a.rows + 7) / 8 * 8 : MAX_ROWS);
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, embed_kernel, a);
}

cudaError_t launch_pe_table(float* pe, int max_ctx, int d, cudaStream_t s) {
    const long long n = (long long)max_ctx * (d / 2);
    pe_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(pe, max_ctx, d);
    return cudaGetLastError();
}

cudaError_t launch_convert_rows(const void* src, int src_bf16, float* dst, int rows, int d, cudaStream_t s) {
    const long long n = (long long)rows * d;
    convert_rows_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(src, src_bf16, dst, n);
    return cudaGetLastError();
}

__global__ void __launch_bounds__(256) save_last_kernel(const float* x, const int* row_seq, const int* row_last,
                                                        float* h_last, int d, unsigned long long* trace) {
    TraceEnd trace_guard(trace);
    pdl_launch_dependents();
    pdl_wait();
    trace_wait(trace);
    const int r = blockIdx.x;
    if (row_seq[r] < 0 || !row_last[r]) return;
    for (int i = threadIdx.x; i < d; i += blockDim.x) h_last[(size_t)row_seq[r] * d + i] = x[(size_t)r * d + i];
}

cudaError_t launch_save_last(const float* x, const int* row_seq, const int* row_last, float* h_last, int d, int rows,
                             unsigned long long* trace, cudaStream_t s, bool pdl) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(rows);
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, save_last_kernel, x, row_seq, row_last, h_last, d, trace);
}

__global__ void trace_reset_kernel(unsigned long long* tr, int records) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= records) return;
    tr[TRACE_WORDS * i] = ~0ull;
    for (int j = 1; j < TRACE_WORDS; ++j) tr[TRACE_WORDS * i + j] = 0;
}

cudaError_t launch_trace_reset(unsigned long long* trace, int records, cudaStream_t s) {
    trace_reset_kernel<<<(records + 255) / 256, 256, 0, s>>>(trace, records);
    return cudaGetLastError();
}

cudaError_t launch_lane_plan(const LanePlanArgs& a, cudaStream_t s, bool pdl) {
    if (a.slots < 1 || a.slots > 1024 || a.rpg < 1 || a.capacity < 1 || a.capacity % a.rpg) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1);
    cfg.blockDim = dim3((a.slots + 31) / 32 * 32);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, lane_plan_kernel, a);
}

cudaError_t launch_slot_set(const SlotSet& set, cudaStream_t s) {
    slot_set_kernel<<<1, 32, 0, s>>>(set);
    return cudaGetLastError();
}

}  // namespace mtp

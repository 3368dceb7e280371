// bsm_topology.cpp -- turns the latency probe into the GB300 stand-in for the
// paper's cluster / memory-bank nearness (Sec. 2.1): which SMs share a die,
// the near and far L2-hit latencies (the Sec. 4.2 weights), and the die of
// each chunk of a buffer (the "bank where a patch is created", Sec. 4.1).
//
// Grouping rule: an SM's latency profile over many lines is high on lines
// homed on the other die and low on its own, so two SMs on one die have
// positively correlated profiles and SMs on different dies negatively
// correlated ones.  SMs are split by the sign of their correlation with the
// first SM seen; a line's home is the group that reaches it faster.  The
// split is accepted only when the correlations are strong and the far
// latency exceeds the near one by at least 5 %.

#include <cuda_runtime.h>

#include <algorithm>
#include <chrono>
#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

#include "bsm_internal.h"

namespace bsm {

constexpr int64_t kProbeBytes = 32ll << 20;
constexpr int kContigLines = 2048;
constexpr int kSpreadLines = 1024;
constexpr int kProbeReps = 8;

namespace {

std::mutex g_topo_mu;
bsm_topology g_topo[64];
bool g_topo_valid[64];

int cuda_fail(cudaError_t e) { return e == cudaSuccess ? BSM_OK : record_cuda_error(e, "topology probe"); }

std::vector<int64_t> default_lines()
{
    std::vector<int64_t> off;
    off.reserve(kContigLines + kSpreadLines);
    for (int i = 0; i < kContigLines; ++i)
        off.push_back(128ll * i);
    for (int k = 0; k < kSpreadLines; ++k)
        off.push_back((1ll << 20) + 30ll * 1024 * k + 128ll * (k % 8));
    return off;
}

}  // namespace

// Raw matrix: lat (host, BSM_MAX_SM x n_lines), seen (host, BSM_MAX_SM).
int probe_latency_host(int device, const std::vector<int64_t> &lines, int reps, std::vector<float> &lat,
                       std::vector<int32_t> &seen)
{
    const int n_lines = static_cast<int>(lines.size());
    if (n_lines <= 0 || reps <= 0 || reps > 1024)
        return BSM_ERR_INVALID_ARG;
    for (int64_t o : lines)
        if (o < 0 || (o & 3) || o + 4 > kProbeBytes)
            return BSM_ERR_INVALID_ARG;
    if (cudaSetDevice(device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    int n_sm = 0;
    if (cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, device) != cudaSuccess)
        return BSM_ERR_CUDA;
    void *buf = nullptr;
    int64_t *d_lines = nullptr;
    float *d_lat = nullptr;
    uint32_t *d_claim = nullptr;
    int rc = BSM_OK;
    const size_t lat_bytes = sizeof(float) * BSM_MAX_SM * (size_t)n_lines;
    do {
        if ((rc = cuda_fail(cudaMalloc(&buf, kProbeBytes))))
            break;
        if ((rc = cuda_fail(cudaMemset(buf, 0, kProbeBytes))))
            break;
        if ((rc = cuda_fail(cudaMalloc(&d_lines, sizeof(int64_t) * n_lines))))
            break;
        if ((rc = cuda_fail(cudaMemcpy(d_lines, lines.data(), sizeof(int64_t) * n_lines,
                                       cudaMemcpyHostToDevice))))
            break;
        if ((rc = cuda_fail(cudaMalloc(&d_lat, lat_bytes))))
            break;
        if ((rc = cuda_fail(cudaMemset(d_lat, 0, lat_bytes))))
            break;
        if ((rc = cuda_fail(cudaMalloc(&d_claim, sizeof(uint32_t) * BSM_MAX_SM))))
            break;
        if ((rc = cuda_fail(cudaMemset(d_claim, 0, sizeof(uint32_t) * BSM_MAX_SM))))
            break;
        if ((rc = cuda_fail(static_cast<cudaError_t>(
                 probe_latency_run(buf, d_lines, n_lines, reps, 8 * n_sm, d_lat, d_claim)))))
            break;
        lat.assign((size_t)BSM_MAX_SM * n_lines, 0.0f);
        std::vector<uint32_t> claim(BSM_MAX_SM, 0);
        if ((rc = cuda_fail(cudaMemcpy(lat.data(), d_lat, lat_bytes, cudaMemcpyDeviceToHost))))
            break;
        if ((rc = cuda_fail(cudaMemcpy(claim.data(), d_claim, sizeof(uint32_t) * BSM_MAX_SM,
                                       cudaMemcpyDeviceToHost))))
            break;
        seen.assign(BSM_MAX_SM, 0);
        for (int s = 0; s < BSM_MAX_SM; ++s)
            seen[s] = claim[s] ? 1 : 0;
    } while (false);
    cudaFree(buf);
    cudaFree(d_lines);
    cudaFree(d_lat);
    cudaFree(d_claim);
    return rc;
}

// Group SMs into dies from the raw matrix (see the file comment).
void analyse_topology(const std::vector<float> &lat, const std::vector<int32_t> &seen, int n_lines,
                      int n_contig, int n_sm, bsm_topology *t)
{
    std::memset(t->sm_die, -1, sizeof(t->sm_die));
    for (int b = 0; b < BSM_MAX_DIES; ++b)
        t->sm_per_die[b] = 0;
    t->n_sm = n_sm;
    t->n_die = 1;
    t->separable = 0;
    t->l_near = t->l_far = 0.0;
    t->separation = 0.0;
    t->granularity = 0;

    std::vector<int> sms;
    for (int s = 0; s < BSM_MAX_SM; ++s)
        if (seen[s])
            sms.push_back(s);
    if (sms.empty())
        return;
    // centred, normalised profile of every SM
    std::vector<std::vector<double>> z(sms.size(), std::vector<double>(n_lines));
    for (size_t k = 0; k < sms.size(); ++k) {
        const float *row = &lat[(size_t)sms[k] * n_lines];
        double mean = 0;
        for (int i = 0; i < n_lines; ++i)
            mean += row[i];
        mean /= n_lines;
        double nrm = 0;
        for (int i = 0; i < n_lines; ++i) {
            z[k][i] = row[i] - mean;
            nrm += z[k][i] * z[k][i];
        }
        nrm = std::sqrt(nrm);
        for (int i = 0; i < n_lines; ++i)
            z[k][i] = nrm > 0 ? z[k][i] / nrm : 0.0;
    }
    std::vector<int> group(sms.size(), 0);
    double sep = 0;
    for (size_t k = 1; k < sms.size(); ++k) {
        double c = 0;
        for (int i = 0; i < n_lines; ++i)
            c += z[k][i] * z[0][i];
        group[k] = c >= 0 ? 0 : 1;
        sep += std::fabs(c);
    }
    sep = sms.size() > 1 ? sep / double(sms.size() - 1) : 0.0;
    int cnt[2] = {0, 0};
    for (int g : group)
        ++cnt[g];
    // per-line mean latency from each group, home = faster group
    std::vector<int> home(n_lines, 0);
    double near_sum = 0, far_sum = 0;
    int used = 0;
    if (cnt[0] > 0 && cnt[1] > 0) {
        for (int i = 0; i < n_lines; ++i) {
            double m[2] = {0, 0};
            for (size_t k = 0; k < sms.size(); ++k)
                m[group[k]] += lat[(size_t)sms[k] * n_lines + i];
            m[0] /= cnt[0];
            m[1] /= cnt[1];
            home[i] = m[0] <= m[1] ? 0 : 1;
            near_sum += std::min(m[0], m[1]);
            far_sum += std::max(m[0], m[1]);
            ++used;
        }
    }
    const double l_near = used ? near_sum / used : 0.0;
    const double l_far = used ? far_sum / used : 0.0;
    t->separation = sep;
    const bool ok = used > 0 && sep >= 0.5 && l_far >= 1.05 * l_near;
    if (!ok) {
        // one "die": every SM seen belongs to it
        double all = 0;
        int n = 0;
        for (int s : sms) {
            t->sm_die[s] = 0;
            for (int i = 0; i < n_lines; ++i) {
                all += lat[(size_t)s * n_lines + i];
                ++n;
            }
        }
        t->sm_per_die[0] = static_cast<int32_t>(sms.size());
        t->l_near = t->l_far = n ? all / n : 0.0;
        t->granularity = 0;
        return;
    }
    t->separable = 1;
    t->n_die = 2;
    t->l_near = l_near;
    t->l_far = l_far;
    for (size_t k = 0; k < sms.size(); ++k) {
        t->sm_die[sms[k]] = static_cast<int8_t>(group[k]);
        ++t->sm_per_die[group[k]];
    }
    // smallest run of same-home lines in the contiguous part
    int64_t best = INT64_MAX;
    int run = 1;
    for (int i = 1; i < n_contig; ++i) {
        if (home[i] == home[i - 1]) {
            ++run;
        } else {
            best = std::min<int64_t>(best, run);
            run = 1;
        }
    }
    t->granularity = best == INT64_MAX ? 128ll * n_contig : 128 * best;
}

int topology_get(int device, int force, bsm_topology *out)
{
    if (device < 0 || device >= 64)
        return BSM_ERR_INVALID_ARG;
    std::lock_guard<std::mutex> lk(g_topo_mu);
    if (g_topo_valid[device] && !force) {
        *out = g_topo[device];
        return BSM_OK;
    }
    int n_sm = 0;
    if (cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    auto t0 = std::chrono::steady_clock::now();
    std::vector<int64_t> lines = default_lines();
    std::vector<float> lat;
    std::vector<int32_t> seen;
    int rc = probe_latency_host(device, lines, kProbeReps, lat, seen);
    if (rc)
        return rc;
    bsm_topology t;
    std::memset(&t, 0, sizeof t);
    t.device = device;
    analyse_topology(lat, seen, static_cast<int>(lines.size()), kContigLines, n_sm, &t);
    t.probe_ms = std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count();
    g_topo[device] = t;
    g_topo_valid[device] = true;
    *out = t;
    return BSM_OK;
}

// The SM -> group table used by the map and the check: the topology's dies,
// or a caller's grouping (entries 0 or 1; -1 = SM not used).
static int group_table(int device, const int8_t *sm_group, int8_t *tab, int *n_sm)
{
    bsm_topology t;
    int rc = topology_get(device, 0, &t);
    if (rc)
        return rc;
    *n_sm = t.n_sm;
    if (!sm_group) {
        if (!t.separable)
            return BSM_ERR_UNSUPPORTED;
        std::memcpy(tab, t.sm_die, BSM_MAX_SM);
        return BSM_OK;
    }
    int cnt[2] = {0, 0};
    for (int s = 0; s < BSM_MAX_SM; ++s) {
        if (sm_group[s] < -1 || sm_group[s] > 1)
            return BSM_ERR_INVALID_ARG;
        tab[s] = sm_group[s];
        if (sm_group[s] >= 0)
            ++cnt[sm_group[s]];
    }
    return cnt[0] > 0 && cnt[1] > 0 ? BSM_OK : BSM_ERR_INVALID_ARG;
}

int addr_die_map_host(int device, const void *ptr, int64_t bytes, int64_t chunk, int8_t *die_out,
                      const int8_t *sm_group)
{
    if (!ptr || !die_out || bytes <= 0 || (bytes & 15) || chunk <= 0 || (chunk & 127) ||
        (reinterpret_cast<uintptr_t>(ptr) & 15))
        return BSM_ERR_INVALID_ARG;
    const int64_t n_chunks = (bytes + chunk - 1) / chunk;
    if (n_chunks > (1ll << 31))
        return BSM_ERR_UNSUPPORTED;
    bsm_topology t;
    int rc = group_table(device, sm_group, t.sm_die, &t.n_sm);
    if (rc)
        return rc;
    if (cudaSetDevice(device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    // every chunk is timed once from an SM of die 0 and once from an SM of
    // die 1; it belongs to the die that reached it faster (ties: alternate)
    float *d_lat = nullptr;
    int8_t *d_sm = nullptr;
    uint32_t *d_ctr = nullptr;
    std::vector<float> lat0, lat1;
    do {
        if ((rc = cuda_fail(cudaMalloc(&d_lat, (size_t)n_chunks * sizeof(float)))))
            break;
        if ((rc = cuda_fail(cudaMalloc(&d_sm, BSM_MAX_SM))))
            break;
        if ((rc = cuda_fail(cudaMemcpy(d_sm, t.sm_die, BSM_MAX_SM, cudaMemcpyHostToDevice))))
            break;
        if ((rc = cuda_fail(cudaMalloc(&d_ctr, sizeof(uint32_t)))))
            break;
        for (int die = 0; die < 2 && !rc; ++die) {
            std::vector<float> &lat = die == 0 ? lat0 : lat1;
            lat.assign(static_cast<size_t>(n_chunks), 0.0f);
            if ((rc = cuda_fail(cudaMemset(d_ctr, 0, sizeof(uint32_t)))))
                break;
            if ((rc = cuda_fail(cudaMemset(d_lat, 0, (size_t)n_chunks * sizeof(float)))))
                break;
            if ((rc = cuda_fail(static_cast<cudaError_t>(
                     probe_map_run(ptr, bytes, chunk, 4, d_sm, die, t.n_sm, d_ctr, d_lat)))))
                break;
            rc = cuda_fail(cudaMemcpy(lat.data(), d_lat, (size_t)n_chunks * sizeof(float), cudaMemcpyDeviceToHost));
        }
        if (rc)
            break;
        for (int64_t c = 0; c < n_chunks; ++c)
            die_out[c] = lat0[c] < lat1[c] ? 0 : (lat1[c] < lat0[c] ? 1 : static_cast<int8_t>(c & 1));
    } while (false);
    cudaFree(d_lat);
    cudaFree(d_sm);
    cudaFree(d_ctr);
    return rc;
}

// Die-map check: the SMs of each die read only the chunks listed for that
// die (the chunks `die_of_chunk` places there, or with invert the others),
// so that a profiler's L2 fabric counters can say how much of the traffic
// still crossed dies.  *xor_out = XOR of every 32-bit word read (each chunk
// is read once: it equals the XOR of the whole buffer).
int die_check_host(int device, const void *ptr, int64_t bytes, int64_t chunk, const int8_t *die_of_chunk,
                   const int8_t *sm_group, int invert, uint32_t *xor_out, float *ms_out)
{
    if (!ptr || !die_of_chunk || !xor_out || bytes <= 0 || chunk <= 0 || (chunk & 15) || bytes % chunk ||
        (reinterpret_cast<uintptr_t>(ptr) & 15))
        return BSM_ERR_INVALID_ARG;
    const int64_t n_chunks = bytes / chunk;
    if (n_chunks >= INT32_MAX || chunk / 16 > INT32_MAX)
        return BSM_ERR_UNSUPPORTED;
    std::vector<int32_t> list[2];
    for (int64_t c = 0; c < n_chunks; ++c) {
        const int d = die_of_chunk[c];
        if (d != 0 && d != 1)
            return BSM_ERR_INVALID_ARG;
        list[invert ? 1 - d : d].push_back(static_cast<int32_t>(c));
    }
    bsm_topology t;
    int rc = group_table(device, sm_group, t.sm_die, &t.n_sm);
    if (rc)
        return rc;
    if (cudaSetDevice(device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    int32_t *d_list = nullptr;
    int8_t *d_sm = nullptr;
    uint32_t *d_words = nullptr;   // two counters, then the XOR sink
    float ms = 0.0f;
    do {
        if ((rc = cuda_fail(cudaMalloc(&d_list, sizeof(int32_t) * static_cast<size_t>(n_chunks)))))
            break;
        if (!list[0].empty() &&
            (rc = cuda_fail(cudaMemcpy(d_list, list[0].data(), sizeof(int32_t) * list[0].size(),
                                       cudaMemcpyHostToDevice))))
            break;
        if (!list[1].empty() &&
            (rc = cuda_fail(cudaMemcpy(d_list + list[0].size(), list[1].data(), sizeof(int32_t) * list[1].size(),
                                       cudaMemcpyHostToDevice))))
            break;
        if ((rc = cuda_fail(cudaMalloc(&d_sm, BSM_MAX_SM))))
            break;
        if ((rc = cuda_fail(cudaMemcpy(d_sm, t.sm_die, BSM_MAX_SM, cudaMemcpyHostToDevice))))
            break;
        if ((rc = cuda_fail(cudaMalloc(&d_words, 4 * sizeof(uint32_t)))))
            break;
        if ((rc = cuda_fail(cudaMemset(d_words, 0, 4 * sizeof(uint32_t)))))
            break;
        if ((rc = cuda_fail(static_cast<cudaError_t>(
                 die_check_run(ptr, n_chunks, chunk, d_list, static_cast<int64_t>(list[0].size()),
                               d_list + list[0].size(), static_cast<int64_t>(list[1].size()), d_words, d_sm,
                               t.n_sm, d_words + 2, &ms)))))
            break;
        rc = cuda_fail(cudaMemcpy(xor_out, d_words + 2, sizeof(uint32_t), cudaMemcpyDeviceToHost));
    } while (false);
    cudaFree(d_list);
    cudaFree(d_sm);
    cudaFree(d_words);
    if (!rc && ms_out)
        *ms_out = ms;
    return rc;
}

}  // namespace bsm
